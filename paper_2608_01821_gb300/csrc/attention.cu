// attention.cu -- bidirectional varlen multi-head attention of one denoising
// step (Sec. 3.1, Eq. 1), on the sm_103a tensor cores.
//
// One persistent CTA per SM (320 threads, warp-specialized).  A work item is
// (request, head, block of up to two 128-row query tiles A and B):
//   warp 8       TMA producer: Q_A and Q_B once per item, then K and V tiles
//                of 128 keys into a 2-stage ring (128-byte swizzle).
//   warp 9       MMA issuer and TMEM owner.  Per key tile j it issues
//                PV_A(j), S_A(j+1), PV_B(j), S_B(j+1), so the tensor pipe
//                works on one tile while the softmax of the other runs.
//   warps 0-3    softmax of tile A, warps 4-7 softmax of tile B: thread r
//                owns query row r; it reads its S row (fp32) from TMEM,
//                keeps the running max in the log2 domain, writes
//                P = 2^(s*c - m) as bf16 back into the first half of its S
//                columns (the PV MMA reads A from TMEM), rescales its O row
//                only when the max grows by more than 2^8 (O and the row sum
//                keep the same stale max, so the result is unchanged) and,
//                after the last key tile, normalizes O and stores it as bf16.
// TMEM: S_A [0,128) S_B [128,256) O_A [256,256+D) O_B [384,384+D).
// Items are ordered longest request first and, within a request,
// head-major, so CTAs running together share a head's K/V in L2.  Keys past
// the end of a request are masked to -inf and their V rows zeroed in shared
// memory, so key tiles may straddle request boundaries and the buffer end.
// With few items (short sequences) one query tile per item is chosen so that
// more SMs get work; when the last of several rounds of two-tile items fills
// at most half of the grid, those items are split into their two tiles.
//
// Fused variant (davet_view_attention, FUSED = true): the step input is never
// packed.  Each request keeps every evidence view as a contiguous block
// [view rows || prompt rows || answer rows] (davet_build_views), so a
// request's sequence for its step view is one run of store rows: every CTA
// derives the requests' view lengths and block starts on the device, and the
// producer loads query, key and value tiles from those runs exactly as the
// packed variant loads them from the packed input.
#include <algorithm>
#include <cstdio>
#include <cstring>
#include <mutex>

#include "common.cuh"

namespace davet {
namespace attn {

constexpr int BM = 128;          // query rows per tile (MMA M)
constexpr int BN = 128;          // keys per tile (N of S = Q K^T, K of O += P V)
constexpr int NS = 2;            // K/V pipeline stages
constexpr int kThreads = 320;    // 2 softmax warpgroups + TMA warp + MMA warp
constexpr int kWarpTma = 8, kWarpMma = 9;
constexpr int kMaxBatch = 1024;  // requests per call
constexpr int kFusedMaxBatch = 256;  // requests per call of the fused variant
constexpr int kMaxLevels = 5;
constexpr int kLptMaxBatch = 256;
constexpr int kChunkBytes = 128 * 128;  // 128 rows x 128 B (64 bf16) swizzled chunk
constexpr uint32_t kTmemCols = 512;
constexpr float kRescaleThreshold = 8.0f;  // log2 units

__host__ __device__ constexpr uint32_t col_s(int t) { return t * 128u; }
__host__ __device__ constexpr uint32_t col_o(int t) { return 256u + t * 128u; }

template <int D, bool FUSED>
struct Smem {
  static constexpr int KC = D / 64;
  static constexpr int kFB = FUSED ? kFusedMaxBatch : 1;
  alignas(1024) uint8_t q[2][KC][kChunkBytes];
  alignas(1024) uint8_t k[NS][KC][kChunkBytes];
  alignas(1024) uint8_t v[NS][KC][kChunkBytes];
  uint64_t q_full, q_empty, fin;
  uint64_t k_full[NS], v_full[NS], k_empty[NS], v_empty[NS];
  uint64_t s_full[2], p_full[2], o_full[2];
  uint32_t tmem;
  int abort;
  int n_req;   // requests with at least one row
  int n_items;
  int n_whole;  // items run with all their query tiles; later ones are halves of two-tile items
  int qtiles;
  int32_t req_start[kMaxBatch];
  int32_t req_len[kMaxBatch];
  int32_t order[kMaxBatch];   // request index of the i-th scheduled request
  int32_t cum[kMaxBatch + 1]; // items before the i-th scheduled request
  // fused variant: first store row of request b's sequence for its view
  int64_t f_base[kFB];
};

struct FusedView {
  long long n_rows;         // rows of the store
  const int64_t* buf_row0;  // first store row of each request's view blocks
  const int32_t* tiles;
  const int32_t* prompt;
  const int32_t* resp;
  const int32_t* level;     // view index per request
  int n_views;
  int rows_per_tile[kMaxLevels + 1];  // view rows per tile of each view
  int32_t* cu_out;
};

struct Params {
  FusedView fv;
  const int32_t* cu;
  int batch;
  int H;
  int max_rows;
  int qtiles;    // query tiles per work item: 1, 2, or 0 = chosen on the device
  int qt2_cost;  // cost of a two-tile item relative to a one-tile item, x16
  float scale_log2;
  uint16_t* out;
  unsigned* err;
};

// Optional timeline trace of CTA 0 (clock64 stamps), compiled in only with
// -DDAVET_ATTN_TRACE for pipeline studies; the product build has none.
#ifdef DAVET_ATTN_TRACE
// region r (0 producer, 1 MMA, 2 softmax A, 3 softmax B) holds 2048 events;
// plain stores only, so recording stays off the critical path
__device__ unsigned long long* g_attn_trace;
// the buffer pointer is read once per role (ATTN_TRACE_DECL), so an event
// costs a clock read and two stores, not a global load
__device__ __forceinline__ void trace_event(unsigned long long* t, unsigned region, unsigned& n, unsigned code,
                                            unsigned idx) {
  if (blockIdx.x != 0 || t == nullptr || n >= 2048) return;
  t[(region * 2048 + n) * 2] = clock64();
  t[(region * 2048 + n) * 2 + 1] = (static_cast<unsigned long long>(code) << 32) | idx;
  ++n;
}
#define ATTN_TRACE(region, code, idx) trace_event(trace_buf, (region), trace_n, (code), (idx))
#define ATTN_TRACE_DECL   \
  unsigned trace_n = 0; \
  unsigned long long* trace_buf = g_attn_trace
#else
#define ATTN_TRACE(region, code, idx) \
  do {                                \
  } while (0)
#define ATTN_TRACE_DECL \
  do {                  \
  } while (0)
#endif

struct Item {
  int b;                              // request
  int start, len, q0, h, nkv, ntile;  // q0: first query row of the item within the request
  int kv0;  // key tile the item starts from (key tiles are visited cyclically)

  // key tile visited at loop step j
  __device__ __forceinline__ int key_tile(int j) const {
    const int k = j + kv0;
    return k >= nkv ? k - nkv : k;
  }
};

// Coordinate along the tensor map's second dimension: slot (0 = query,
// 1 = key, 2 = value) of head h.
__device__ __forceinline__ int h_coord(int slot, int h, int H) { return slot * H + h; }

template <typename S>
__device__ __forceinline__ Item decode(const S& s, int item, int H, int qtiles) {
  // items from n_whole on are the two halves (one query tile each) of the
  // last round's two-tile items
  int half = -1;
  if (item >= s.n_whole) {
    const int k = item - s.n_whole;
    item = s.n_whole + (k >> 1);
    half = k & 1;
  }
  // largest i with cum[i] <= item
  int lo = 0, hi = s.n_req - 1;
  while (lo < hi) {
    const int mid = (lo + hi + 1) >> 1;
    if (s.cum[mid] <= item) lo = mid; else hi = mid - 1;
  }
  const int b = s.order[lo];
  const int local = item - s.cum[lo];
  const int len = s.req_len[b];
  const int shift = qtiles == 2 ? 8 : 7;  // log2 of the rows per item
  const int rows_per_item = 1 << shift;
  const int nq = (len + rows_per_item - 1) >> shift;
  Item it;
  it.b = b;
  it.start = s.req_start[b];
  it.len = len;
  it.h = local / nq;
  it.q0 = (local - it.h * nq) * rows_per_item;
  it.nkv = (len + BN - 1) / BN;
  // query blocks of one head start at evenly spread key tiles, so CTAs that
  // run together on the same head read different K/V lines at any moment
  const int qb = local - it.h * nq;
  // (32-bit division when the product fits: a 64-bit one is a long
  // subroutine, and every role decodes every item)
  const long long qk = static_cast<long long>(qb) * it.nkv;
  it.kv0 = qk < 0x7fffffffLL ? static_cast<int>(static_cast<unsigned>(qk) / static_cast<unsigned>(nq))
                             : static_cast<int>(qk / nq);
  it.ntile = (qtiles == 2 && it.q0 + BM < len) ? 2 : 1;
  if (half >= 0) {
    // a half whose tile lies past the request end computes rows it never stores
    it.q0 += half * BM;
    it.ntile = 1;
  }
  return it;
}

// All lanes wait; the outcome is made warp-uniform.
__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, unsigned* err, volatile int* abort_flag) {
  const bool ok = mbar_wait(bar, parity, err, abort_flag);
  return __all_sync(0xffffffffu, ok);
}

template <int D, bool FUSED>
__global__ void __launch_bounds__(kThreads, 1)
    attention_kernel(const __grid_constant__ CUtensorMap tmap, Params prm) {
  constexpr int KC = D / 64;
  extern __shared__ uint8_t smem_raw[];
  using SM = Smem<D, FUSED>;
  SM& s = *reinterpret_cast<SM*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const FusedView& fv = prm.fv;

  const int tid = threadIdx.x;
  const int warp = tid >> 5;
  const int lane = tid & 31;
  const int H = prm.H;

  // ------------------------------------ barriers, TMEM (no global memory)
  if (tid == 0) {
    s.abort = 0;
    mbar_init(&s.q_full, 1);
    mbar_init(&s.q_empty, 1);
    mbar_init(&s.fin, 1);
    for (int i = 0; i < NS; ++i) {
      mbar_init(&s.k_full[i], 1);
      mbar_init(&s.v_full[i], 1);
      mbar_init(&s.k_empty[i], 1);
      mbar_init(&s.v_empty[i], 1);
    }
    for (int t = 0; t < 2; ++t) {
      mbar_init(&s.s_full[t], 1);
      mbar_init(&s.p_full[t], 128);
      mbar_init(&s.o_full[t], 1);
    }
    fence_mbar_init();
  }
  if (warp == kWarpMma) {
    tmem_alloc(&s.tmem, kTmemCols);
    tmem_relinquish();
  }
  if (warp == kWarpTma && lane == 0) tma_prefetch_desc(&tmap);
  pdl_launch_dependents();
  pdl_wait();  // cu_seqlens and qkv come from the previous kernel

  // ---------------------------------------------------------- schedule
  if (FUSED && tid == 0) {
    // view lengths and packed starts, as davet_gather_view computes them, and
    // where each request's sequence starts in the store: its view block
    bool bad = false;
    long long run = 0;
    int n = 0;
    for (int b = 0; b < prm.batch; ++b) {
      const int v = fv.level[b], nt = fv.tiles[b], pl = fv.prompt[b], rl = fv.resp[b];
      long long nvis = 0, base = fv.buf_row0[b];
      const long long text = static_cast<long long>(max(pl, 0)) + max(rl, 0);
      if (v < 0 || v >= fv.n_views || nt < 0 || pl < 0 || rl < 0) {
        bad = true;
        base = -1;
      } else {
        for (int u = 0; u < v; ++u) base += static_cast<long long>(nt) * fv.rows_per_tile[u] + text;
        nvis = static_cast<long long>(nt) * fv.rows_per_tile[v];
      }
      const long long len = base >= 0 ? nvis + text : 0;
      if (base >= 0 && base + len > fv.n_rows) bad = true;  // rows past the store read as zeros
      const long long a = min(run, static_cast<long long>(prm.max_rows));
      const long long e = min(run + len, static_cast<long long>(prm.max_rows));
      run += len;
      s.req_start[b] = static_cast<int32_t>(a);
      s.req_len[b] = static_cast<int32_t>(e - a);
      s.f_base[b] = base;
      if (e > a) s.order[n++] = b;
      if (blockIdx.x == 0) fv.cu_out[b] = static_cast<int32_t>(a);
    }
    if (blockIdx.x == 0) {
      fv.cu_out[prm.batch] = static_cast<int32_t>(min(run, static_cast<long long>(prm.max_rows)));
      if (bad) raise_error(prm.err, DEV_ERR_ARG);
      if (run > prm.max_rows) raise_error(prm.err, DEV_ERR_CAPACITY);
    }
    s.n_req = n;
  }
  if (!FUSED && tid == 0) {
    bool bad = false;
    int prev_end = 0;
    int n = 0;
    for (int b = 0; b < prm.batch; ++b) {
      int a = prm.cu[b], e = prm.cu[b + 1];
      if (a < prev_end || a > prm.max_rows || e < a || e > prm.max_rows) bad = true;
      a = min(max(a, prev_end), prm.max_rows);
      e = min(max(e, a), prm.max_rows);
      prev_end = e;
      s.req_start[b] = a;
      s.req_len[b] = e - a;
      if (e > a) s.order[n++] = b;
    }
    if (bad && blockIdx.x == 0) raise_error(prm.err, DEV_ERR_ARG);
    s.n_req = n;
  }
  __syncthreads();
  // longest request first (stable); only for modest batches (one request
  // is already in order)
  if (s.n_req > 1 && s.n_req <= kLptMaxBatch) {
    int my_b = -1, my_rank = 0;
    if (tid < s.n_req) {
      my_b = s.order[tid];
      const int L = s.req_len[my_b];
      for (int j = 0; j < s.n_req; ++j) {
        const int bj = s.order[j];
        const int Lj = s.req_len[bj];
        my_rank += (Lj > L) || (Lj == L && bj < my_b);
      }
    }
    __syncthreads();
    if (tid < s.n_req) s.order[my_rank] = my_b;
    __syncthreads();
  }
  if (tid == 0) {
    // query tiles per item: two tiles keep the tensor pipe busy while the
    // other tile's softmax runs, one tile gives more items when sequences
    // are short; pick the smaller estimated makespan (rounds of items over
    // the grid, an item with two tiles costing qt2_cost/16 of a one-tile item)
    int qt = prm.qtiles;
    if (qt == 0) {
      long long i1 = 0, i2 = 0;
      for (int i = 0; i < s.n_req; ++i) {
        const int L = s.req_len[s.order[i]];
        i1 += (L + BM - 1) / BM;
        i2 += (L + 2 * BM - 1) / (2 * BM);
      }
      const long long g = gridDim.x;
      if (i1 * H <= g) {
        qt = 1;  // one round of one-tile items: two tiles cannot take fewer rounds
      } else {
        // rounds of items over the grid (32-bit division when the counts
        // fit: a 64-bit one is a long subroutine on the path every CTA waits for)
        auto rounds = [g](long long n) -> long long {
          return n < 0x7fffffffLL ? static_cast<long long>((static_cast<unsigned>(n) + static_cast<unsigned>(g) - 1u) /
                                                           static_cast<unsigned>(g))
                                  : (n + g - 1) / g;
        };
        const long long c1 = rounds(i1 * H) * 16;
        const long long c2 = rounds(i2 * H) * prm.qt2_cost;
        qt = c2 <= c1 ? 2 : 1;
      }
    }
    s.qtiles = qt;
    int acc = 0;
    const int rows_per_item = BM * qt;
    for (int i = 0; i < s.n_req; ++i) {
      s.cum[i] = acc;
      acc += ((s.req_len[s.order[i]] + rows_per_item - 1) / rows_per_item) * H;
    }
    s.cum[s.n_req] = acc;
    // when the last of several rounds of two-tile items fills at most half of
    // the grid, its items run as two one-tile items each (on twice as many
    // CTAs), so the launch ends after a one-tile item rather than a two-tile one
    int split = 0;
    const int g = static_cast<int>(gridDim.x);
    if (qt == 2 && acc > g) {
      const int r = acc % g;
      if (r > 0 && 2 * r <= g) split = r;
    }
    s.n_whole = acc - split;
    s.n_items = acc + split;
  }
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s.tmem;
  const int qtiles = s.qtiles;
  volatile int* abort_flag = &s.abort;

  if (warp == kWarpTma) {
    // ------------------------------------------------------ TMA producer
    // rows of the item's request: packed input (cu) or its view block
    if (lane == 0) {
      ATTN_TRACE_DECL;
      uint32_t it = 0, wi = 0, nq = 0, nk = 0, nv = 0;  // loads issued (query tiles, K, V)
      bool ok = true;
      for (int item = blockIdx.x; ok && item < s.n_items; item += gridDim.x, ++wi) {
        const Item w = decode(s, item, H, qtiles);
        const long long src0 = FUSED ? s.f_base[w.b] : w.start;
        if (wi > 0) ok = mbar_wait(&s.q_empty, (wi - 1) & 1, prm.err, abort_flag);
        if (!ok) break;
        mbar_arrive_expect_tx(&s.q_full, w.ntile * KC * kChunkBytes);
        for (int t = 0; t < w.ntile; ++t)
          for (int c = 0; c < KC; ++c)
            tma_load_3d(s.q[t][c], &tmap, &s.q_full, 64 * c, h_coord(0, w.h, H), src0 + w.q0 + t * BM);
        ++nq;
        for (int j = 0; j < w.nkv; ++j, ++it) {
          const int st = it % NS;
          const int row = static_cast<int>(src0 + w.key_tile(j) * BN);
          // K of stage st is free once the S MMAs of the tile that used it completed
          if (it >= NS) ok = mbar_wait(&s.k_empty[st], ((it / NS) - 1) & 1, prm.err, abort_flag);
          if (!ok) break;
          ATTN_TRACE(0, 2, it);
          mbar_arrive_expect_tx(&s.k_full[st], KC * kChunkBytes);
          for (int c = 0; c < KC; ++c) tma_load_3d(s.k[st][c], &tmap, &s.k_full[st], 64 * c, h_coord(1, w.h, H), row);
          ++nk;
          // V of stage st is free once the PV MMAs of that tile completed
          if (it >= NS) ok = mbar_wait(&s.v_empty[st], ((it / NS) - 1) & 1, prm.err, abort_flag);
          if (!ok) break;
          mbar_arrive_expect_tx(&s.v_full[st], KC * kChunkBytes);
          for (int c = 0; c < KC; ++c) tma_load_3d(s.v[st][c], &tmap, &s.v_full[st], 64 * c, h_coord(2, w.h, H), row);
          ++nv;
          ATTN_TRACE(0, 1, it);
        }
      }
      if (!ok) {
        // let copies already in flight land before the CTA exits: the last
        // query tiles (the MMA warp may not have waited for them) and the
        // last NS key and NS value tiles issued
        if (nq > 0) mbar_wait(&s.q_full, (nq - 1) & 1, nullptr, nullptr);
        for (uint32_t i = (nk > NS ? nk - NS : 0); i < nk; ++i) mbar_wait(&s.k_full[i % NS], (i / NS) & 1, nullptr, nullptr);
        for (uint32_t i = (nv > NS ? nv - NS : 0); i < nv; ++i) mbar_wait(&s.v_full[i % NS], (i / NS) & 1, nullptr, nullptr);
      }
    }
  } else if (warp == kWarpMma) {
    // --------------------------------------------------------- MMA issuer
    // One thread issues every MMA.  tcgen05.mma issue is sensitive to the code
    // around it (a branch between two MMAs starves the tensor pipe), so each
    // group of D/16 or BN/16 MMAs is straight-line code with precomputed
    // descriptors and immediate accumulate flags.
    if (lane == 0) {
      ATTN_TRACE_DECL;
      constexpr uint32_t kIdescQK = idesc_bf16_f32(BM, BN, false, false);
      constexpr uint32_t kIdescPV = idesc_bf16_f32(BM, D, false, true);
      // only the start-address field (16-byte units) differs between MMAs
      const uint64_t q_desc0 = sw128_desc(smem_u32(s.q[0][0]), 16, 1024);
      const uint64_t k_desc0 = sw128_desc(smem_u32(s.k[0][0]), 16, 1024);
      const uint64_t v_desc0 = sw128_desc(smem_u32(s.v[0][0]), kChunkBytes, 1024);
      constexpr uint32_t kTile16 = (KC * kChunkBytes) >> 4;  // one Q tile / K or V stage
      uint32_t it = 0, wi = 0;
      uint32_t np[2] = {0, 0};  // P tiles consumed per query tile
      bool ok = true;

      // S_t = Q_t K^T for the K tile in stage st
      auto issue_s = [&](int t, int st) {
        const uint64_t a0 = q_desc0 + t * kTile16;
        const uint64_t b0 = k_desc0 + st * kTile16;
        const uint32_t d = tmem + col_s(t);
        umma_ss_imm<false>(d, a0, b0, kIdescQK);
#pragma unroll
        for (int kk = 1; kk < D / 16; ++kk) {
          const uint32_t off = ((kk >> 2) * kChunkBytes + (kk & 3) * 32) >> 4;
          umma_ss_imm<true>(d, a0 + off, b0 + off, kIdescQK);
        }
        umma_commit(&s.s_full[t]);
      };
      // O_t (+)= P_t V for the V tile in stage st, P read from TMEM
      auto issue_pv = [&](int t, int st, bool first) {
        const uint64_t b0 = v_desc0 + st * kTile16;
        const uint32_t d = tmem + col_o(t);
        const uint32_t a = tmem + col_s(t);
        if (first)
          umma_ts_imm<false>(d, a, b0, kIdescPV);
        else
          umma_ts_imm<true>(d, a, b0, kIdescPV);
#pragma unroll
        for (int kk = 1; kk < BN / 16; ++kk) umma_ts_imm<true>(d, a + kk * 8, b0 + kk * (2048 >> 4), kIdescPV);
      };

      for (int item = blockIdx.x; ok && item < s.n_items; item += gridDim.x, ++wi) {
        const Item w = decode(s, item, H, qtiles);
        ok = mbar_wait(&s.q_full, wi & 1, prm.err, abort_flag);
        if (!ok) break;
        // prologue: S for key tile 0
        ok = mbar_wait(&s.k_full[it % NS], (it / NS) & 1, prm.err, abort_flag);
        if (!ok) break;
        tc_fence_after();
        issue_s(0, it % NS);
        if (w.ntile == 2) issue_s(1, it % NS);
        umma_commit(&s.k_empty[it % NS]);
        if (w.nkv == 1) umma_commit(&s.q_empty);
        for (int j = 0; j < w.nkv; ++j, ++it) {
          const int st = it % NS;
          const int st1 = (it + 1) % NS;
          const bool more = j + 1 < w.nkv;
          ok = mbar_wait(&s.v_full[st], (it / NS) & 1, prm.err, abort_flag);
          if (!ok) break;
          ATTN_TRACE(1, 10, it);
          // tile A: PV, then S of the next key tile
          ok = mbar_wait(&s.p_full[0], np[0] & 1, prm.err, abort_flag);
          if (!ok) break;
          ATTN_TRACE(1, 12, it);
          ++np[0];
          tc_fence_after();
          issue_pv(0, st, j == 0);
          // the V stage is released with the next commits (after S, when
          // there is a next key tile): a commit alone between two MMA groups
          // leaves the tensor pipe idle for a while
          if (more) {
            ok = mbar_wait(&s.k_full[st1], ((it + 1) / NS) & 1, prm.err, abort_flag);
            if (!ok) break;
              ATTN_TRACE(1, 11, it);
            tc_fence_after();
            issue_s(0, st1);
            if (w.ntile == 1) {
              umma_commit(&s.v_empty[st]);
              umma_commit(&s.k_empty[st1]);
              if (j + 1 == w.nkv - 1) umma_commit(&s.q_empty);
            }
          } else {
            if (w.ntile == 1) umma_commit(&s.v_empty[st]);
            umma_commit(&s.o_full[0]);
          }
          if (w.ntile == 2) {
            // tile B: PV, then S of the next key tile
            ok = mbar_wait(&s.p_full[1], np[1] & 1, prm.err, abort_flag);
            if (!ok) break;
            ATTN_TRACE(1, 13, it);
            ++np[1];
            tc_fence_after();
            issue_pv(1, st, j == 0);
            if (more) {
              issue_s(1, st1);
              umma_commit(&s.v_empty[st]);
              umma_commit(&s.k_empty[st1]);
              if (j + 1 == w.nkv - 1) umma_commit(&s.q_empty);
            } else {
              umma_commit(&s.v_empty[st]);
              umma_commit(&s.o_full[1]);
            }
          }
        }
      }
      // wait until every issued MMA has completed before TMEM is released
      umma_commit(&s.fin);
      mbar_wait(&s.fin, 0, nullptr, nullptr);
    }
  } else {
    // ------------------------------------------------- softmax + epilogue
    const int t = warp >> 2;             // query tile of this warpgroup
    const int r = tid & 127;             // query row within the tile == TMEM lane
    const uint32_t lane_base = static_cast<uint32_t>((warp & 3) * 32) << 16;
    const uint32_t s_addr = tmem + lane_base + col_s(t);
    const uint32_t o_addr = tmem + lane_base + col_o(t);
    ATTN_TRACE_DECL;
    const float c = prm.scale_log2;
    uint32_t ns = 0, no = 0;
    bool ok = true;
    for (int item = blockIdx.x; ok && item < s.n_items; item += gridDim.x) {
      const Item w = decode(s, item, H, qtiles);
      if (t >= w.ntile) continue;
      float m = -INFINITY;  // running max of c * score (log2 domain)
      float l = 0.f;        // running sum of 2^(c*score - m)
      for (int j = 0; j < w.nkv; ++j, ++ns) {
        ok = warp_wait(&s.s_full[t], ns & 1, prm.err, abort_flag);
        if (!ok) break;
        if (r == 0) ATTN_TRACE(2 + t, 20 + t, ns);
        tc_fence_after();
        // all four TMEM loads in flight before one wait
        // the row in two halves: the second half's TMEM load is in flight
        // while the first half's max is taken
        uint32_t raw[BN];
        tmem_ld32(s_addr, *reinterpret_cast<uint32_t(*)[32]>(&raw[0]));
        tmem_ld32(s_addr + 32, *reinterpret_cast<uint32_t(*)[32]>(&raw[32]));
        tmem_wait_ld_regs(&raw[0]);
        tmem_ld32(s_addr + 64, *reinterpret_cast<uint32_t(*)[32]>(&raw[64]));
        tmem_ld32(s_addr + 96, *reinterpret_cast<uint32_t(*)[32]>(&raw[96]));
        if (r == 0) ATTN_TRACE(2 + t, 22 + t, ns);
        float* x = reinterpret_cast<float*>(raw);
        const int valid = min(BN, w.len - w.key_tile(j) * BN);
        if (t == 0 && valid < BN) {
          // keys past the request end: zero their V rows before PV reads them
          // (P is 0 there, but the rows may hold anything, including
          // non-finite values).  Tile A's key-tile count equals the global
          // key-tile counter, so ns names the V stage and phase.
          ok = warp_wait(&s.v_full[ns % NS], (ns / NS) & 1, prm.err, abort_flag);
          if (!ok) break;
          if (r >= valid) {
#pragma unroll
            for (int cc = 0; cc < KC; ++cc) {
              uint4* row = reinterpret_cast<uint4*>(s.v[ns % NS][cc] + r * 128);
#pragma unroll
              for (int u = 0; u < 8; ++u) row[u] = make_uint4(0, 0, 0, 0);
            }
          }
          fence_proxy_async_smem();
        }
        if (valid < BN / 2) {
#pragma unroll
          for (int i = 0; i < BN / 2; ++i) x[i] = (i < valid) ? x[i] : -INFINITY;
        }
        // row max: eight independent chains of three-input max, then a tree
        float mp[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) mp[u] = fmaxf(x[u], x[u + 8]);
#pragma unroll
        for (int i = 16; i < BN / 2; i += 16)
#pragma unroll
          for (int u = 0; u < 8; ++u) mp[u] = fmax3(mp[u], x[i + u], x[i + 8 + u]);
        tmem_wait_ld_regs(&raw[64]);
        if (valid < BN) {
#pragma unroll
          for (int i = BN / 2; i < BN; ++i) x[i] = (i < valid) ? x[i] : -INFINITY;
        }
#pragma unroll
        for (int i = BN / 2; i < BN; i += 16)
#pragma unroll
          for (int u = 0; u < 8; ++u) mp[u] = fmax3(mp[u], x[i + u], x[i + 8 + u]);
        const float mx = fmax3(fmax3(mp[0], mp[1], mp[2]), fmax3(mp[3], mp[4], mp[5]), fmaxf(mp[6], mp[7]));
        if (r == 0) ATTN_TRACE(2 + t, 26 + t, ns);
        const float mt = mx * c;
        float factor = 1.f;
        bool need = false;
        if (j == 0) {
          m = mt;
        } else if (mt > m + kRescaleThreshold) {
          factor = ex2(m - mt);
          m = mt;
          need = true;
        }
        const float neg_m = -m;
        // p = 2^(c*s - m): packed FMA for two scores, two SFU exponentials,
        // rounded to bf16.  The row sum adds the rounded weights, the values
        // the PV MMA multiplies V by, so the weights applied to V sum to one
        // after the final division (four accumulators).
        float rsum[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int q = 0; q < BN / 32; ++q) {
          uint32_t pk[16];
#pragma unroll
          for (int i = 0; i < 16; ++i) {
            float a0, a1;
            ffma2(a0, a1, x[32 * q + 2 * i], x[32 * q + 2 * i + 1], c, c, neg_m, neg_m);
            pk[i] = pack_bf16x2(ex2(a0), ex2(a1));
            const int h = (i & 1) * 2;
            add_bf16x2_f32(rsum[h], rsum[h + 1], pk[i]);
          }
          tmem_st16(s_addr + 16 * q, pk);
        }
        const float rs = (rsum[0] + rsum[1]) + (rsum[2] + rsum[3]);
        if (r == 0) ATTN_TRACE(2 + t, 28 + t, ns);
        // O is settled here (S of this tile was issued after the previous
        // PV of this tile) and no MMA touches it before P is published
        if (j > 0 && __any_sync(0xffffffffu, need)) {
          uint32_t o[32];
#pragma unroll 1
          for (int q = 0; q < D / 32; ++q) {
            tmem_ld32(o_addr + 32 * q, o);
            tmem_wait_ld();
#pragma unroll
            for (int i = 0; i < 32; ++i) o[i] = __float_as_uint(__uint_as_float(o[i]) * factor);
            tmem_st32(o_addr + 32 * q, o);
          }
        }
        l = (j == 0) ? rs : l * factor + rs;
        tmem_wait_st();
        tc_fence_before();
        mbar_arrive(&s.p_full[t]);
        if (r == 0) ATTN_TRACE(2 + t, 24 + t, ns);
      }
      if (!ok) break;
      // ------------------------------------------------------- epilogue
      ok = warp_wait(&s.o_full[t], no & 1, prm.err, abort_flag);
      ++no;
      if (!ok) break;
      tc_fence_after();
      const float inv_l = 1.f / l;
      const int qrow = w.q0 + t * BM + r;
      const bool row_ok = qrow < w.len;
      uint16_t* dst = prm.out + (static_cast<int64_t>(w.start + qrow) * H + w.h) * D;
#pragma unroll
      for (int q = 0; q < D / 32; ++q) {
        uint32_t o[32];
        tmem_ld32(o_addr + 32 * q, o);
        tmem_wait_ld();
        if (row_ok) {
          uint4* d4 = reinterpret_cast<uint4*>(dst + 32 * q);
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            uint4 v;
            v.x = pack_bf16x2(__uint_as_float(o[8 * u + 0]) * inv_l, __uint_as_float(o[8 * u + 1]) * inv_l);
            v.y = pack_bf16x2(__uint_as_float(o[8 * u + 2]) * inv_l, __uint_as_float(o[8 * u + 3]) * inv_l);
            v.z = pack_bf16x2(__uint_as_float(o[8 * u + 4]) * inv_l, __uint_as_float(o[8 * u + 5]) * inv_l);
            v.w = pack_bf16x2(__uint_as_float(o[8 * u + 6]) * inv_l, __uint_as_float(o[8 * u + 7]) * inv_l);
            d4[u] = v;
          }
        }
      }
      tc_fence_before();
    }
  }

  // ------------------------------------------------------------ teardown
  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

}  // namespace attn

namespace {

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn get_encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
            cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
  });
  return fn;
}

struct DeviceInfo {
  int sms = 0;
  bool attr_set[4] = {false, false, false, false};
};
DeviceInfo g_dev[64];
std::mutex g_dev_mu;

// Launches the packed variant (FUSED = false: qkv is the packed input, cu its
// boundaries) or the fused one (FUSED = true: qkv is the row store of view
// blocks, fv describes the requests; cu is unused).
template <int D, bool FUSED>
davet_status launch(const void* qkv, const int32_t* cu, const attn::FusedView& fv, int batch, int64_t max_rows, int H,
                    float scale, void* out, cudaStream_t stream) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  if (dev < 0 || dev >= 64) return DAVET_ERR_UNSUPPORTED;
  const size_t smem = sizeof(attn::Smem<D, FUSED>) + 1024;
  {
    std::lock_guard<std::mutex> g(g_dev_mu);
    DeviceInfo& di = g_dev[dev];
    if (di.sms == 0) {
      e = cudaDeviceGetAttribute(&di.sms, cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess) return cuda_fail(e);
    }
    const int slot = (D == 128 ? 1 : 0) + (FUSED ? 2 : 0);
    if (!di.attr_set[slot]) {
      e = cudaFuncSetAttribute(attn::attention_kernel<D, FUSED>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               static_cast<int>(smem));
      if (e != cudaSuccess) return cuda_fail(e);
      di.attr_set[slot] = true;
    }
  }
  unsigned* err = device_error_word();
  if (!err) return DAVET_ERR_CUDA;
  EncodeTiledFn enc = get_encode_fn();
  if (!enc) return DAVET_ERR_CUDA;
  // packed variant: the packed input; fused: the row store of view blocks
  CUtensorMap tmap;
  const int64_t map_rows = FUSED ? fv.n_rows : max_rows;
  const cuuint64_t gdim[3] = {static_cast<cuuint64_t>(D), static_cast<cuuint64_t>(3 * H),
                              static_cast<cuuint64_t>(std::max<int64_t>(map_rows, 1))};
  const cuuint64_t gstride[2] = {static_cast<cuuint64_t>(D) * 2, static_cast<cuuint64_t>(3) * H * D * 2};
  const cuuint32_t box[3] = {64, 1, 128};
  const cuuint32_t estride[3] = {1, 1, 1};
  CUresult cr = enc(&tmap, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(qkv), gdim, gstride, box, estride,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS) return DAVET_ERR_INVALID_ARG;

  attn::Params prm;
  prm.fv = fv;
  prm.cu = cu;
  prm.batch = batch;
  prm.H = H;
  prm.max_rows = static_cast<int>(max_rows);
  prm.qtiles = 0;
  prm.qt2_cost = 24;
  if (const char* e = std::getenv("DAVET_ATTN_QTILES")) prm.qtiles = std::atoi(e) == 1 ? 1 : (std::atoi(e) == 2 ? 2 : 0);
  prm.scale_log2 = static_cast<float>(static_cast<double>(scale) * 1.4426950408889634);
  prm.out = static_cast<uint16_t*>(out);
  prm.err = err;

  const int64_t items_bound = ((max_rows + attn::BM - 1) / attn::BM + batch) * static_cast<int64_t>(H);
  const int grid = static_cast<int>(std::min<int64_t>(items_bound, g_dev[dev].sms));
  if (grid <= 0) return DAVET_OK;
  e = davet::launch(attn::attention_kernel<D, FUSED>, dim3(grid), dim3(attn::kThreads), smem, stream, tmap, prm);
  return e == cudaSuccess ? DAVET_OK : cuda_fail(e);
}

}  // namespace
}  // namespace davet

#ifdef DAVET_ATTN_TRACE
extern "C" int davet_debug_attn_trace(void* buf) {
  unsigned long long* p = static_cast<unsigned long long*>(buf);
  return static_cast<int>(cudaMemcpyToSymbol(davet::attn::g_attn_trace, &p, sizeof p));
}
#endif

extern "C" davet_status davet_step_attention(const void* qkv, const int32_t* cu_seqlens_dev, int batch,
                                             int64_t max_total_rows, int H, int D, float scale, void* out,
                                             void* stream) {
  using namespace davet;
  if (batch < 0 || max_total_rows < 0 || H < 1 || !(scale > 0.f)) return DAVET_ERR_INVALID_ARG;
  if (batch == 0 || max_total_rows == 0) return DAVET_OK;
  if (!qkv || !cu_seqlens_dev || !out) return DAVET_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(qkv) | reinterpret_cast<uintptr_t>(out)) & 15u) return DAVET_ERR_INVALID_ARG;
  if (D != 64 && D != 128) return DAVET_ERR_UNSUPPORTED;
  if (batch > attn::kMaxBatch) return DAVET_ERR_UNSUPPORTED;
  if (max_total_rows > (int64_t(1) << 30) || static_cast<int64_t>(3) * H > 65535) return DAVET_ERR_UNSUPPORTED;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const attn::FusedView none{};
  return D == 128 ? launch<128, false>(qkv, cu_seqlens_dev, none, batch, max_total_rows, H, scale, out, st)
                  : launch<64, false>(qkv, cu_seqlens_dev, none, batch, max_total_rows, H, scale, out, st);
}

extern "C" davet_status davet_view_attention(const void* store, int64_t store_rows, const int64_t* buf_row0_dev,
                                             const int32_t* tiles_dev, const int32_t* prompt_len_dev,
                                             const int32_t* resp_len_dev, const int32_t* view_dev, int batch,
                                             int grid, int n_levels, int mixed_level, int mixed_stride, int H, int D,
                                             float scale, void* out, int32_t* cu_seqlens_dev, int64_t max_total_rows,
                                             void* stream) {
  using namespace davet;
  if (batch < 0 || max_total_rows < 0 || H < 1 || !(scale > 0.f) || store_rows < 0) return DAVET_ERR_INVALID_ARG;
  int rpt[attn::kMaxLevels + 1];
  int n_views = 0;
  const davet_status ls = davet_view_rows(grid, n_levels, mixed_level, mixed_stride, rpt, &n_views);
  if (ls != DAVET_OK) return ls;
  if (D != 64 && D != 128) return DAVET_ERR_UNSUPPORTED;
  if (batch > attn::kFusedMaxBatch) return DAVET_ERR_UNSUPPORTED;
  if (max_total_rows > (int64_t(1) << 30) || static_cast<int64_t>(3) * H > 65535) return DAVET_ERR_UNSUPPORTED;
  if (store_rows > 0x7fffffffLL) return DAVET_ERR_UNSUPPORTED;
  if (!cu_seqlens_dev) return DAVET_ERR_INVALID_ARG;
  if (batch == 0) return DAVET_OK;
  if (!store || !buf_row0_dev || !tiles_dev || !prompt_len_dev || !resp_len_dev || !view_dev || !out)
    return DAVET_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(store) | reinterpret_cast<uintptr_t>(out)) & 15u) return DAVET_ERR_INVALID_ARG;
  attn::FusedView fv{};
  fv.n_rows = store_rows;
  fv.buf_row0 = buf_row0_dev;
  fv.tiles = tiles_dev;
  fv.prompt = prompt_len_dev;
  fv.resp = resp_len_dev;
  fv.level = view_dev;
  fv.n_views = n_views;
  for (int v = 0; v <= attn::kMaxLevels; ++v) fv.rows_per_tile[v] = v < n_views ? rpt[v] : 0;
  fv.cu_out = cu_seqlens_dev;
  if (max_total_rows == 0) return DAVET_OK;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  return D == 128 ? launch<128, true>(store, nullptr, fv, batch, max_total_rows, H, scale, out, st)
                  : launch<64, true>(store, nullptr, fv, batch, max_total_rows, H, scale, out, st);
}
