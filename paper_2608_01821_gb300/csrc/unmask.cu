// unmask.cu -- confidence-ranked commitment of one denoising step (Sec. 3.1,
// Eq. 1-2) and the step statistics that feed the trajectory risk (Eq. 7).
//
// Two kernels:
//  1. row kernel: every (answer row, vocabulary chunk of 8 or 16 KB) is one
//     warp.
//     A warp of a masked row streams its chunk of bf16 logits once with 128-bit
//     loads (eight in flight per lane) and keeps, per lane, an online
//     (max, sum of 2^(x*log2e - max*log2e), first argmax) triple, merged by
//     shuffles and written to the workspace.  Independent warps keep many
//     loads in flight per SM and hide each other's latencies.
//  2. select: one CTA per request.  Each thread combines one row's chunk
//     triples (stored chunk-major, so the loads coalesce; one round of
//     loads) into (argmax, conf = 1/sum) held in shared memory, counting
//     churn against the previous argmax; after one barrier, warp 0 forms
//     the mean confidence and takes the top-k rows by (conf desc, position
//     asc) with k rounds of a warp arg-max, and commits them.
// Both kernels are latency-bound at small sizes: a dependent round trip to
// L2 costs about half a microsecond here, so every load a kernel needs is
// issued in one batch, without branches between the loads.

#include <algorithm>
#include <climits>
#include <mutex>

#include "common.cuh"

namespace davet {
namespace unm {

constexpr int kRowThreads = 256;  // 8 warps, one (row, chunk) unit each
constexpr int kMaxChunks = 64;
constexpr int kLoads = 8;         // 16-byte loads in flight per lane
// The select runs 512 threads combining records in rounds of 16 when a row
// has at most 16 chunks (one round of loads each; a 512-row request in one
// pass), else 256 threads with rounds of 32 (the register budget of a
// 32-record round allows 256 threads).
constexpr int kSelThreadsNarrow = 512, kSelGroupNarrow = 16;
constexpr int kSelThreadsWide = 256, kSelGroupWide = 32;
constexpr int kSelSmemRows = 4096;
constexpr float kLog2e = 1.4426950408889634f;

struct __align__(16) Partial {
  float m;    // max logit (raw, bf16-exact)
  float s;    // sum of 2^(x*log2e - m*log2e)
  int idx;    // first index attaining the max
  int pad;
};

struct Layout {
  int nchunk;  // vocabulary chunks per row (one warp each)
  size_t off_partial, off_conf, off_idx, bytes;
};

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

// Chunks of 1024 slices (16 KB: four rounds of loads per lane) when the
// call has at least kWideUnits such (row, chunk) units, which is enough to
// keep every SM streaming, else of 512 slices (8 KB), so that few answer rows
// still spread over many warps; at most kMaxChunks per row.  Longer chunks
// mean fewer blocks per call (a late step, with few rows still masked, pays
// for launching the blocks of every row) and fewer records for the select to
// combine.  When `max_bytes` is given (the allocation-free path), fewer and
// longer chunks so that the layout fits.  The conf / argmax arrays serve
// requests longer than kSelSmemRows rows.
constexpr int64_t kWideUnits = 8192;
inline Layout layout_for(int64_t total_rows, int V, size_t max_bytes = ~size_t(0)) {
  Layout L;
  const int64_t v8 = V / 8;
  const size_t rows = static_cast<size_t>(total_rows);
  const size_t fixed = align256(rows * sizeof(float)) + align256(rows * sizeof(int32_t));
  const int64_t slices = total_rows * ((v8 + 1023) / 1024) >= kWideUnits ? 1024 : 512;
  int64_t nchunk = std::max<int64_t>(1, std::min<int64_t>(kMaxChunks, (v8 + slices - 1) / slices));
  while (nchunk > 1 && align256(rows * nchunk * sizeof(Partial)) + fixed > max_bytes) --nchunk;
  L.nchunk = static_cast<int>(nchunk);
  L.off_partial = 0;
  L.off_conf = align256(rows * L.nchunk * sizeof(Partial));
  L.off_idx = L.off_conf + align256(rows * sizeof(float));
  L.bytes = L.off_idx + align256(rows * sizeof(int32_t));
  return L;
}

// 2^x on the SFU; not volatile, so the compiler may interleave it
__device__ __forceinline__ float sfu_ex2(float x) {
  float y;
  asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
  return y;
}

__device__ __forceinline__ uint32_t max_bf16x2(uint32_t a, uint32_t b) {
  uint32_t r;
  asm("max.bf16x2 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(b));
  return r;
}

// Warp-wide combination of the lanes' triples in two passes instead of
// pairwise merges: the warp max M by shuffles, one rescale 2^((m - M)log2e)
// per lane, then a shuffle sum and the smallest index among lanes at M.
// Every lane returns the result.
__device__ __forceinline__ Partial warp_combine(Partial p) {
  float mx = p.m;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
  float sm = p.s > 0.f ? __fmul_rn(p.s, sfu_ex2((p.m - mx) * kLog2e)) : 0.f;
  int ix = p.m == mx ? p.idx : INT_MAX;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    sm += __shfl_xor_sync(0xffffffffu, sm, o);
    ix = min(ix, __shfl_xor_sync(0xffffffffu, ix, o));
  }
  Partial r;
  r.m = mx;
  r.s = sm;
  r.idx = ix;
  r.pad = 0;
  return r;
}

__device__ __forceinline__ Partial empty_partial() {
  Partial p;
  p.m = -INFINITY;
  p.s = 0.f;
  p.idx = INT_MAX;
  p.pad = 0;
  return p;
}

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// A lane's running state: max m (raw), m * log2e, first argmax, and the sum
// of 2^(x*log2e - m*log2e) in two accumulators (one per element parity).
struct Run {
  float m, ml, s0, s1;
  int idx;
};

__device__ __forceinline__ Run empty_run() {
  Run r;
  r.m = -INFINITY;
  r.ml = -INFINITY;
  r.s0 = 0.f;
  r.s1 = 0.f;
  r.idx = INT_MAX;
  return r;
}

// Fold one 16-byte slice (8 logits starting at vocabulary index w0) into r:
// the slice's max comes from packed bf16 maxima; only a new running max
// (rare after the first slices) takes the branch that finds its first
// index and rescales the sums.  Each pair of terms costs one packed FMA,
// two SFU exponentials and one packed add.
__device__ __forceinline__ void fold(Run& r, uint4 u, int w0) {
  const uint32_t mx = max_bf16x2(max_bf16x2(u.x, u.y), max_bf16x2(u.z, u.w));
  const float vm = fmaxf(bf16lo(mx), bf16hi(mx));
  if (vm > r.m) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
    int first = 7;
#pragma unroll
    for (int k = 7; k >= 0; --k) {
      const float xk = (k & 1) ? bf16hi(w[k >> 1]) : bf16lo(w[k >> 1]);
      first = (xk == vm) ? k : first;
    }
    r.idx = w0 + first;
    // explicit roundings: no contraction into an FMA, which could differ
    // between the kernels this is inlined into
    const float ml = __fmul_rn(vm, kLog2e);
    const float f = r.s0 + r.s1 > 0.f ? sfu_ex2(__fsub_rn(r.ml, ml)) : 0.f;
    r.s0 *= f;
    r.s1 *= f;
    r.m = vm;
    r.ml = ml;
  }
  const float nm = -r.ml;
  float a[8];
  ffma2(a[0], a[1], bf16lo(u.x), bf16hi(u.x), kLog2e, kLog2e, nm, nm);
  ffma2(a[2], a[3], bf16lo(u.y), bf16hi(u.y), kLog2e, kLog2e, nm, nm);
  ffma2(a[4], a[5], bf16lo(u.z), bf16hi(u.z), kLog2e, kLog2e, nm, nm);
  ffma2(a[6], a[7], bf16lo(u.w), bf16hi(u.w), kLog2e, kLog2e, nm, nm);
  float e[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) e[k] = sfu_ex2(a[k]);
  float t0, t1, t2, t3;
  fadd2(t0, t1, e[0], e[1], e[2], e[3]);
  fadd2(t2, t3, e[4], e[5], e[6], e[7]);
  fadd2(t0, t1, t0, t1, t2, t3);
  fadd2(r.s0, r.s1, r.s0, r.s1, t0, t1);
}

// Fold a lane's batch of kLoads slices: u[m] holds the 8 logits from
// vocabulary index w0 + 256 m (the lane's slices of one piece, 32 slices
// apart).  The batch's max is found first, by one tree of packed bf16 maxima,
// so the running max, its first index and the rescale are updated at most
// once per batch (first index: lowest m, then lowest position in the
// slice); the terms of every slice are then summed as in fold, relative to
// the batch's running max.
__device__ __forceinline__ void fold_batch(Run& r, const uint4 (&u)[kLoads], int w0) {
  uint32_t sm[kLoads];
#pragma unroll
  for (int m = 0; m < kLoads; ++m) sm[m] = max_bf16x2(max_bf16x2(u[m].x, u[m].y), max_bf16x2(u[m].z, u[m].w));
  uint32_t t[kLoads / 2];
#pragma unroll
  for (int m = 0; m < kLoads / 2; ++m) t[m] = max_bf16x2(sm[2 * m], sm[2 * m + 1]);
  const uint32_t bm = max_bf16x2(max_bf16x2(t[0], t[1]), max_bf16x2(t[2], t[3]));
  const float vm = fmaxf(bf16lo(bm), bf16hi(bm));
  if (vm > r.m) {
    // the first slice holding vm, then its first position
    uint32_t w[4] = {0u, 0u, 0u, 0u};
    int fm = 0;
#pragma unroll
    for (int m = kLoads - 1; m >= 0; --m) {
      if (fmaxf(bf16lo(sm[m]), bf16hi(sm[m])) == vm) {
        fm = m;
        w[0] = u[m].x;
        w[1] = u[m].y;
        w[2] = u[m].z;
        w[3] = u[m].w;
      }
    }
    int first = 7;
#pragma unroll
    for (int k = 7; k >= 0; --k) {
      const float xk = (k & 1) ? bf16hi(w[k >> 1]) : bf16lo(w[k >> 1]);
      first = (xk == vm) ? k : first;
    }
    r.idx = w0 + 256 * fm + first;
    // explicit roundings: no contraction into an FMA, which could differ
    // between the kernels this is inlined into
    const float ml = __fmul_rn(vm, kLog2e);
    const float f = r.s0 + r.s1 > 0.f ? sfu_ex2(__fsub_rn(r.ml, ml)) : 0.f;
    r.s0 *= f;
    r.s1 *= f;
    r.m = vm;
    r.ml = ml;
  }
  const float nm = -r.ml;
#pragma unroll
  for (int m = 0; m < kLoads; ++m) {
    float a[8];
    ffma2(a[0], a[1], bf16lo(u[m].x), bf16hi(u[m].x), kLog2e, kLog2e, nm, nm);
    ffma2(a[2], a[3], bf16lo(u[m].y), bf16hi(u[m].y), kLog2e, kLog2e, nm, nm);
    ffma2(a[4], a[5], bf16lo(u[m].z), bf16hi(u[m].z), kLog2e, kLog2e, nm, nm);
    ffma2(a[6], a[7], bf16lo(u[m].w), bf16hi(u[m].w), kLog2e, kLog2e, nm, nm);
    float e[8];
#pragma unroll
    for (int k = 0; k < 8; ++k) e[k] = sfu_ex2(a[k]);
    float t0, t1, t2, t3;
    fadd2(t0, t1, e[0], e[1], e[2], e[3]);
    fadd2(t2, t3, e[4], e[5], e[6], e[7]);
    fadd2(t0, t1, t0, t1, t2, t3);
    fadd2(r.s0, r.s1, r.s0, r.s1, t0, t1);
  }
}

__device__ __forceinline__ Partial to_partial(const Run& r) {
  Partial p;
  p.m = r.m;
  p.s = r.s0 + r.s1;
  p.idx = r.idx;
  p.pad = 0;
  return p;
}

struct RowArgs {
  const uint4* logits;
  int V8;
  int nchunk;
  int chunk;  // 16-byte slices per chunk
  long long total_rows;
  const uint8_t* masked;
  Partial* partial;  // [nchunk][rows]
};

__global__ void __launch_bounds__(kRowThreads) row_kernel(RowArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  const long long unit = (static_cast<long long>(blockIdx.x) * kRowThreads + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (unit >= a.total_rows * a.nchunk) return;
  // unit < 2^31 (rows and chunks are bounded on the host): a 32-bit division
  const unsigned u32 = static_cast<unsigned>(unit);
  const long long row = u32 / static_cast<unsigned>(a.nchunk);
  if (!a.masked[row]) return;
  const int ch = static_cast<int>(u32 - static_cast<unsigned>(row) * static_cast<unsigned>(a.nchunk));
  const int lo = ch * a.chunk, hi = min(a.V8, lo + a.chunk);
  const uint4* base = a.logits + row * static_cast<long long>(a.V8);
  Run run = empty_run();
  // every load of an iteration is issued before the first fold
  for (int v = lo + lane; v < hi; v += 32 * kLoads) {
    uint4 u[kLoads];
#pragma unroll
    for (int k = 0; k < kLoads; ++k)
      if (v + 32 * k < hi) u[k] = ld_stream(base + v + 32 * k);
    if (v + 32 * (kLoads - 1) < hi) {
      fold_batch(run, u, v * 8);
    } else {
#pragma unroll
      for (int k = 0; k < kLoads; ++k)
        if (v + 32 * k < hi) fold(run, u[k], (v + 32 * k) * 8);
    }
  }
  const Partial p = warp_combine(to_partial(run));
  // chunk-major, so the select's row-per-thread loads are coalesced
  if (lane == 0) a.partial[static_cast<long long>(ch) * a.total_rows + row] = p;
}

struct SelArgs {
  const Partial* partial;
  int nchunk;
  const int32_t* cu;
  int batch;
  long long total_rows;
  int k;
  uint8_t* masked;
  int32_t* tokens;
  int32_t* argmax;
  float* conf_out;
  int32_t* committed;
  float* stats;
  float* row_conf;   // workspace for requests longer than kSelSmemRows
  int32_t* row_idx;
  unsigned* err;
};

// Warp arg-max of (conf, -pos): the winning (conf, pos) on every lane.
__device__ __forceinline__ void warp_best(float& c, int& pos) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float c2 = __shfl_xor_sync(0xffffffffu, c, o);
    const int p2 = __shfl_xor_sync(0xffffffffu, pos, o);
    if (c2 > c || (c2 == c && p2 < pos)) {
      c = c2;
      pos = p2;
    }
  }
}

// Combination of chunks [c0, min(c0 + G, nc)) of one row's triples in two
// passes: the max M, then the sum of s * 2^((m - M)log2e) and the smallest
// index among chunks at M.
template <int G>
__device__ __forceinline__ Partial combine_group(const Partial* __restrict__ part, long long rows, long long i, int c0,
                                                 int nc) {
  float m[G], sv[G];
  int ix[G];
#pragma unroll
  for (int c = 0; c < G; ++c) {
    const bool ok = c0 + c < nc;
    const Partial v = part[static_cast<long long>(ok ? c0 + c : 0) * rows + i];
    m[c] = ok ? v.m : -INFINITY;
    sv[c] = ok ? v.s : 0.f;
    ix[c] = ok ? v.idx : INT_MAX;
  }
  float mx = m[0];
#pragma unroll
  for (int c = 1; c < G; ++c) mx = fmaxf(mx, m[c]);
  Partial r;
  r.m = mx;
  r.s = 0.f;
  r.idx = INT_MAX;
  r.pad = 0;
#pragma unroll
  for (int c = 0; c < G; ++c) {
    if (sv[c] > 0.f) r.s += sv[c] * sfu_ex2((m[c] - mx) * kLog2e);
    if (m[c] == mx) r.idx = min(r.idx, ix[c]);
  }
  return r;
}

// (argmax, conf) of one row from all its chunk triples.
template <int G>
__device__ __forceinline__ void combine_row(const Partial* __restrict__ part, long long rows, long long i, int nc,
                                            float& conf, int& idx) {
  Partial p = combine_group<G>(part, rows, i, 0, nc);
  for (int c0 = G; c0 < nc; c0 += G) {
    const Partial q = combine_group<G>(part, rows, i, c0, nc);
    const float mx = fmaxf(p.m, q.m);
    const float sp = p.s > 0.f ? p.s * sfu_ex2((p.m - mx) * kLog2e) : 0.f;
    const float sq = q.s > 0.f ? q.s * sfu_ex2((q.m - mx) * kLog2e) : 0.f;
    p.idx = p.m == mx ? (q.m == mx ? min(p.idx, q.idx) : p.idx) : q.idx;
    p.m = mx;
    p.s = sp + sq;
  }
  conf = 1.f / p.s;
  idx = p.idx == INT_MAX ? 0 : p.idx;
}

// One CTA per request.  Each thread combines one row's chunk triples per
// pass (one round of coalesced loads); after one barrier, warp 0 forms the
// statistics and takes the top-k with k rounds of a warp arg-max over the
// rows' confidences in shared memory.
template <int kSelThreads, int kGroup>
__global__ void __launch_bounds__(kSelThreads) select_kernel(SelArgs a) {
  __shared__ float s_conf_buf[kSelSmemRows];
  __shared__ int32_t s_idx_buf[kSelSmemRows];
  __shared__ float s_sum[kSelThreads / 32];
  __shared__ int s_cnt[3][kSelThreads / 32];
  pdl_launch_dependents();
  pdl_wait();
  const int b = blockIdx.x;
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  constexpr int kWarps = kSelThreads / 32;
  const long long cu0 = a.cu[b], cu1 = a.cu[b + 1];
  const long long s0 = min(max(cu0, 0LL), a.total_rows);
  const long long s1 = min(max(cu1, s0), a.total_rows);
  if (tid == 0 && (cu0 != s0 || cu1 != s1)) raise_error(a.err, DEV_ERR_ARG);
  const long long n = s1 - s0;
  // per-row results: shared memory when the request fits, else workspace;
  // conf = -3 marks a row that is not masked (or already committed)
  float* cbuf = n <= kSelSmemRows ? s_conf_buf : a.row_conf + s0;
  int32_t* ibuf = n <= kSelSmemRows ? s_idx_buf : a.row_idx + s0;

  // the mask, the previous argmax and the chunk triples of a row are loaded
  // together (triples of unmasked rows are stale and discarded)
  float conf_sum = 0.f;
  int n_masked = 0, n_both = 0, n_changed = 0;
  for (long long r = tid; r < n; r += kSelThreads) {
    const long long i = s0 + r;
    const uint8_t m8 = a.masked[i];
    const int prev = a.argmax ? a.argmax[i] : -1;
    float conf;
    int idx;
    combine_row<kGroup>(a.partial, a.total_rows, i, a.nchunk, conf, idx);
    if (!m8) {
      cbuf[r] = -3.f;
      continue;
    }
    cbuf[r] = conf;
    ibuf[r] = idx;
    if (a.conf_out) a.conf_out[i] = conf;
    if (a.argmax) a.argmax[i] = idx;
    conf_sum += conf;
    ++n_masked;
    if (prev >= 0) {
      ++n_both;
      n_changed += prev != idx;
    }
  }
  // block sums in a fixed order: a shuffle tree per warp, then warps in order
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    conf_sum += __shfl_xor_sync(0xffffffffu, conf_sum, o);
    n_masked += __shfl_xor_sync(0xffffffffu, n_masked, o);
    n_both += __shfl_xor_sync(0xffffffffu, n_both, o);
    n_changed += __shfl_xor_sync(0xffffffffu, n_changed, o);
  }
  if (lane == 0) {
    s_sum[warp] = conf_sum;
    s_cnt[0][warp] = n_masked;
    s_cnt[1][warp] = n_both;
    s_cnt[2][warp] = n_changed;
  }
  __syncthreads();
  if (warp != 0) return;

  float tot_conf = 0.f;
  int tot_masked = 0, tot_both = 0, tot_changed = 0;
#pragma unroll
  for (int w = 0; w < kWarps; ++w) {
    tot_conf += s_sum[w];
    tot_masked += s_cnt[0][w];
    tot_both += s_cnt[1][w];
    tot_changed += s_cnt[2][w];
  }
  if (lane == 0 && a.stats) {
    a.stats[2 * b + 0] = tot_masked ? tot_conf / static_cast<float>(tot_masked) : 0.f;
    a.stats[2 * b + 1] = tot_both ? static_cast<float>(tot_changed) / static_cast<float>(tot_both) : 0.f;
  }
  // top-k: k rounds of a warp arg-max over the rows still masked
  const int take = min(a.k, tot_masked);
  int j = 0;
  // (positions in 32 bits: a request has fewer than 2^31 rows)
  const int n32 = static_cast<int>(n);
  for (; j < take; ++j) {
    float best_c = -2.f;
    int best_pos = INT_MAX;
    for (int i = lane; i < n32; i += 32) {
      const float c = cbuf[i];
      if (c > best_c || (c == best_c && i < best_pos)) {
        best_c = c;
        best_pos = i;
      }
    }
    const int mine = best_pos;
    warp_best(best_c, best_pos);
    if (best_pos == INT_MAX) break;  // only when confidences are not numbers
    if (mine == best_pos) {
      a.tokens[s0 + best_pos] = ibuf[best_pos];
      a.masked[s0 + best_pos] = 0;
      cbuf[best_pos] = -3.f;
      if (a.committed) a.committed[static_cast<long long>(b) * a.k + j] = static_cast<int32_t>(best_pos);
    }
    __syncwarp();
  }
  if (a.committed)
    for (int q = j + lane; q < a.k; q += 32) a.committed[static_cast<long long>(b) * a.k + q] = -1;
}

// The row pass with bulk copies: each warp's (row, chunk) unit arrives in
// 4 KB pieces through the copy engine of the SM (cp.async.bulk into shared
// memory, two pieces in flight per warp), not through L1, then folds from
// shared memory.  Each lane folds the same elements in the same order as in
// row_kernel, so the results are bit-identical.
constexpr int kPiece = 256;  // 16-byte slices per bulk piece (4 KB)
static_assert(kPiece == 32 * kLoads, "a lane's slices of a piece are one batch of row_kernel");

struct RowStage {  // one warp's two pieces and their barriers
  uint4 buf[2][kPiece];
  uint64_t bar[2];
};
constexpr size_t kRowBulkSmem = sizeof(RowStage) * (kRowThreads / 32);

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes, uint64_t* bar) {
  asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
               ::"r"(smem_u32(dst)), "l"(src), "r"(bytes), "r"(smem_u32(bar))
               : "memory");
}

__global__ void __launch_bounds__(kRowThreads) row_kernel_bulk(RowArgs a, unsigned* err) {
  extern __shared__ __align__(128) uint8_t row_smem[];
  RowStage* ws = reinterpret_cast<RowStage*>(row_smem) + (threadIdx.x >> 5);
  const int lane = threadIdx.x & 31;
  if (lane == 0) {
    mbar_init(&ws->bar[0], 1);
    mbar_init(&ws->bar[1], 1);
    fence_mbar_init();
  }
  __syncwarp();
  pdl_launch_dependents();
  pdl_wait();
  const long long unit = (static_cast<long long>(blockIdx.x) * kRowThreads + threadIdx.x) >> 5;
  if (unit >= a.total_rows * a.nchunk) return;
  // unit < 2^31 (rows and chunks are bounded on the host): a 32-bit division
  const unsigned u32 = static_cast<unsigned>(unit);
  const long long row = u32 / static_cast<unsigned>(a.nchunk);
  if (!a.masked[row]) return;
  const int ch = static_cast<int>(u32 - static_cast<unsigned>(row) * static_cast<unsigned>(a.nchunk));
  const int lo = ch * a.chunk, hi = min(a.V8, lo + a.chunk);
  const int n = hi - lo;
  const int npieces = (n + kPiece - 1) / kPiece;
  const uint4* src = a.logits + row * static_cast<long long>(a.V8) + lo;
  auto issue = [&](int p) {  // lane 0
    const int sl = p & 1;
    const int cnt = min(kPiece, n - p * kPiece);
    mbar_arrive_expect_tx(&ws->bar[sl], static_cast<uint32_t>(cnt) * 16u);
    bulk_g2s(&ws->buf[sl][0], src + p * kPiece, static_cast<uint32_t>(cnt) * 16u, &ws->bar[sl]);
  };
  if (lane == 0) {
    issue(0);
    if (npieces > 1) issue(1);
  }
  Run run = empty_run();
  int p = 0;
  for (; p < npieces; ++p) {
    const int sl = p & 1;
    const bool ok = __all_sync(0xffffffffu, mbar_wait(&ws->bar[sl], (p >> 1) & 1, err, nullptr));
    if (!ok) break;
    const int cnt = min(kPiece, n - p * kPiece);
    const int w0 = (lo + p * kPiece) * 8;
    // the lane's slices of the piece are those of one plain-load iteration
    // of row_kernel, folded the same way (bit-identical results)
    if (lane + 32 * (kLoads - 1) < cnt) {
      uint4 u[kLoads];
#pragma unroll
      for (int m = 0; m < kLoads; ++m) u[m] = ws->buf[sl][lane + 32 * m];
      fold_batch(run, u, w0 + lane * 8);
    } else {
      for (int k = lane; k < cnt; k += 32) fold(run, ws->buf[sl][k], w0 + k * 8);
    }
    __syncwarp();
    if (lane == 0 && p + 2 < npieces) {
      fence_proxy_async_smem();  // the warp's reads of this piece before the copy's writes
      issue(p + 2);
    }
  }
  if (p < npieces) {
    // a wait gave up: let the copies still in flight land before the warp
    // leaves (bounded), and write nothing
    if (lane == 0)
      for (int q = p; q < min(npieces, p + 2); ++q) mbar_wait(&ws->bar[q & 1], (q >> 1) & 1, nullptr, nullptr);
    return;
  }
  const Partial pt = warp_combine(to_partial(run));
  // chunk-major, so the select's row-per-thread loads are coalesced
  if (lane == 0) a.partial[static_cast<long long>(ch) * a.total_rows + row] = pt;
}

// Whether p is device memory (the bulk row pass reads only device memory;
// pinned host memory mapped for the device takes the plain-load pass).
inline bool device_memory(const void* p) {
  cudaPointerAttributes at;
  if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
    (void)cudaGetLastError();
    return false;
  }
  return at.type == cudaMemoryTypeDevice;
}

// The bulk row pass's dynamic shared memory limit, once per device.
inline cudaError_t set_row_bulk_smem() {
  static std::mutex mu;
  static bool done[64] = {};
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return e;
  if (dev < 0 || dev >= 64) return cudaErrorInvalidDevice;
  std::lock_guard<std::mutex> g(mu);
  if (done[dev]) return cudaSuccess;
  e = cudaFuncSetAttribute(row_kernel_bulk, cudaFuncAttributeMaxDynamicSharedMemorySize,
                           static_cast<int>(kRowBulkSmem));
  if (e == cudaSuccess) done[dev] = true;
  return e;
}

// Both kernels of one call on `stream`, over the workspace `ws` (layout L).
inline davet_status enqueue(const void* logits, int V, const int32_t* cu, int batch, int64_t total_rows, int k,
                            uint8_t* masked, int32_t* tokens, int32_t* argmax, float* conf, int32_t* committed,
                            float* stats, uint8_t* ws, const Layout& L, cudaStream_t stream) {
  unsigned* err = device_error_word();
  if (!err) return DAVET_ERR_CUDA;
  Partial* partial = reinterpret_cast<Partial*>(ws + L.off_partial);
  if (total_rows > 0) {
    RowArgs r;
    r.logits = static_cast<const uint4*>(logits);
    r.V8 = V / 8;
    r.nchunk = L.nchunk;
    r.chunk = (r.V8 + L.nchunk - 1) / L.nchunk;
    r.total_rows = total_rows;
    r.masked = masked;
    r.partial = partial;
    const long long warps = total_rows * L.nchunk;
    const long long blocks = (warps + kRowThreads / 32 - 1) / (kRowThreads / 32);
    cudaError_t e;
    if (device_memory(logits)) {
      e = set_row_bulk_smem();
      if (e == cudaSuccess)
        e = launch(row_kernel_bulk, dim3(static_cast<unsigned>(blocks)), dim3(kRowThreads), kRowBulkSmem, stream, r,
                   err);
    } else {
      // host-mapped logits: plain loads
      e = launch(row_kernel, dim3(static_cast<unsigned>(blocks)), dim3(kRowThreads), 0, stream, r);
    }
    if (e != cudaSuccess) return cuda_fail(e);
  }
  SelArgs a;
  a.partial = partial;
  a.nchunk = L.nchunk;
  a.cu = cu;
  a.batch = batch;
  a.total_rows = total_rows;
  a.k = k;
  a.masked = masked;
  a.tokens = tokens;
  a.argmax = argmax;
  a.conf_out = conf;
  a.committed = committed;
  a.stats = stats;
  a.row_conf = reinterpret_cast<float*>(ws + L.off_conf);
  a.row_idx = reinterpret_cast<int32_t*>(ws + L.off_idx);
  a.err = err;
  const cudaError_t e =
      L.nchunk <= kSelGroupNarrow
          ? launch(select_kernel<kSelThreadsNarrow, kSelGroupNarrow>, dim3(batch), dim3(kSelThreadsNarrow), 0, stream, a)
          : launch(select_kernel<kSelThreadsWide, kSelGroupWide>, dim3(batch), dim3(kSelThreadsWide), 0, stream, a);
  return e == cudaSuccess ? DAVET_OK : cuda_fail(e);
}

}  // namespace unm
}  // namespace davet

extern "C" davet_status davet_unmask_topk_workspace(int64_t total_rows, int V, int batch, size_t* bytes) {
  if (total_rows < 0 || V < 8 || V % 8 != 0 || batch < 0 || !bytes) return DAVET_ERR_INVALID_ARG;
  *bytes = davet::unm::layout_for(total_rows, V).bytes;
  return DAVET_OK;
}

extern "C" davet_status davet_unmask_topk(const void* logits, int V, const int32_t* cu_resp_dev, int batch,
                                          int64_t total_rows, int k, uint8_t* masked_dev, int32_t* tokens_dev,
                                          int32_t* argmax_dev, float* conf_dev, int32_t* committed_dev,
                                          float* stats_dev, void* workspace, size_t workspace_bytes, void* stream) {
  using namespace davet;
  using namespace davet::unm;
  if (batch < 0 || total_rows < 0 || V < 8 || V % 8 != 0 || k < 1 || k > 1024) return DAVET_ERR_INVALID_ARG;
  if (batch == 0) return DAVET_OK;
  if (!cu_resp_dev || !masked_dev || !tokens_dev) return DAVET_ERR_INVALID_ARG;
  if (total_rows > 0 && (!logits || !workspace)) return DAVET_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(logits) & 15u) return DAVET_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(workspace) & 255u) return DAVET_ERR_INVALID_ARG;
  if (batch > 65535 || total_rows > (int64_t(1) << 31) / 64) return DAVET_ERR_UNSUPPORTED;
  const Layout L = layout_for(total_rows, V);
  if (total_rows > 0 && workspace_bytes < L.bytes) return DAVET_ERR_INVALID_ARG;
  return enqueue(logits, V, cu_resp_dev, batch, total_rows, k, masked_dev, tokens_dev, argmax_dev, conf_dev,
                 committed_dev, stats_dev, static_cast<uint8_t*>(workspace), L, static_cast<cudaStream_t>(stream));
}

// ---------------------------------------------------------------------------
// Staging of the rows the unmasking will read: row i of `src` (device
// addressable: device memory or pinned host memory) is copied to row i of
// `dst` wherever masked[i] != 0.  One warp per (row, 16 KB chunk), eight
// 16-byte loads per lane issued before their stores.
namespace davet {
namespace unm {

__global__ void __launch_bounds__(kRowThreads) stage_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst,
                                                            int V8, int nchunk, int chunk, long long total_rows,
                                                            const uint8_t* __restrict__ masked) {
  pdl_launch_dependents();
  pdl_wait();
  const long long unit = (static_cast<long long>(blockIdx.x) * kRowThreads + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (unit >= total_rows * nchunk) return;
  // unit < 2^31 (rows and chunks are bounded on the host): a 32-bit division
  const unsigned u32 = static_cast<unsigned>(unit);
  const long long row = u32 / static_cast<unsigned>(nchunk);
  if (!masked[row]) return;
  const int ch = static_cast<int>(u32 - static_cast<unsigned>(row) * static_cast<unsigned>(nchunk));
  const int lo = ch * chunk, hi = min(V8, lo + chunk);
  const uint4* s = src + row * static_cast<long long>(V8);
  uint4* d = dst + row * static_cast<long long>(V8);
  for (int v = lo + lane; v < hi; v += 32 * kLoads) {
    uint4 u[kLoads];
#pragma unroll
    for (int k = 0; k < kLoads; ++k)
      if (v + 32 * k < hi) u[k] = ld_stream(s + v + 32 * k);
#pragma unroll
    for (int k = 0; k < kLoads; ++k)
      if (v + 32 * k < hi) d[v + 32 * k] = u[k];
  }
}

}  // namespace unm
}  // namespace davet

extern "C" davet_status davet_stage_masked_rows(const void* src, int V, const uint8_t* masked_dev, int64_t total_rows,
                                                void* dst, void* stream) {
  using namespace davet;
  using namespace davet::unm;
  if (V < 8 || V % 8 != 0 || total_rows < 0) return DAVET_ERR_INVALID_ARG;
  if (total_rows == 0) return DAVET_OK;
  if (!src || !dst || !masked_dev) return DAVET_ERR_INVALID_ARG;
  if ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15u) return DAVET_ERR_INVALID_ARG;
  if (total_rows > (int64_t(1) << 31) / 64) return DAVET_ERR_UNSUPPORTED;
  const int V8 = V / 8;
  // 16 KB per warp: over the host link fewer, longer streams do better
  // than 8 KB chunks (4, 8, 16, 32, 64 KB and whole rows measured)
  const int nchunk = std::max(1, std::min(kMaxChunks, (V8 + 1023) / 1024));
  const int chunk = (V8 + nchunk - 1) / nchunk;
  const long long warps = total_rows * nchunk;
  const long long blocks = (warps + kRowThreads / 32 - 1) / (kRowThreads / 32);
  const cudaError_t e = launch(stage_kernel, dim3(static_cast<unsigned>(blocks)), dim3(kRowThreads), 0,
                               static_cast<cudaStream_t>(stream), static_cast<const uint4*>(src),
                               static_cast<uint4*>(dst), V8, nchunk, chunk, static_cast<long long>(total_rows),
                               masked_dev);
  if (e != cudaSuccess) return cuda_fail(e);
  return check_launch();
}

// ---------------------------------------------------------------------------
// Allocation-free variant of davet_unmask_topk.
//
// Its scratch lives in a fixed device array owned by the library, so the
// caller passes only inputs and outputs.  Every device that loads the library
// keeps this array for the life of the process, and all calls on a device
// share it.  Nothing in it needs clearing: the select reads only the
// triples of masked rows, which the row kernel of the same call writes.
namespace davet {
namespace unm {

constexpr size_t kNoAllocScratchBytes = size_t(1) << 20;  // DAVET_NOALLOC_SCRATCH_BYTES
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kNoAllocMaxDevices = 64;

// The array's device address, kept per device together with the unique id
// of the CUDA context it was looked up in (0: none yet).
struct NoAllocAddr {
  unsigned long long ctx_id;
  uint8_t* ptr;
};
static NoAllocAddr g_noalloc_addr[kNoAllocMaxDevices] = {};
static std::mutex g_noalloc_mu;

using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

// Unique id of the calling thread's current context, 0 when there is none
// yet (the runtime creates the primary context at its first device call).
static unsigned long long current_ctx_id() {
  static CtxGetCurrentFn get_current = nullptr;
  static CtxGetIdFn get_id = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_current = reinterpret_cast<CtxGetCurrentFn>(p);
    p = nullptr;
    if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      get_id = reinterpret_cast<CtxGetIdFn>(p);
  });
  CUcontext ctx = nullptr;
  unsigned long long id = 0;
  if (!get_current || !get_id || get_current(&ctx) != CUDA_SUCCESS || !ctx) return 0;
  if (get_id(ctx, &id) != CUDA_SUCCESS) return 0;
  return id;
}

// Device address of g_noalloc_scratch in the current context.  Host code only
// sees a host-side stand-in for the array under its name, so the address is
// asked for with the device current, once per context, and kept.
static uint8_t* noalloc_scratch(davet_status* st) {
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) {
    *st = cuda_fail(e);
    return nullptr;
  }
  if (dev < 0 || dev >= kNoAllocMaxDevices) {
    *st = DAVET_ERR_UNSUPPORTED;
    return nullptr;
  }
  std::lock_guard<std::mutex> g(g_noalloc_mu);
  NoAllocAddr& a = g_noalloc_addr[dev];
  const unsigned long long id = current_ctx_id();
  if (id == 0 || a.ctx_id != id || !a.ptr) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) {
      *st = cuda_fail(e);
      return nullptr;
    }
    a.ptr = static_cast<uint8_t*>(p);
    // the look-up made the context current if there was none
    a.ctx_id = current_ctx_id();
  }
  return a.ptr;
}

}  // namespace unm
}  // namespace davet

extern "C" davet_status davet_unmask_topk_noalloc(const void* logits, int V, const int32_t* cu_resp_dev, int batch,
                                                  int64_t total_rows, int k, uint8_t* masked_dev,
                                                  int32_t* tokens_dev, int32_t* argmax_dev, float* conf_dev,
                                                  int32_t* committed_dev, float* stats_dev, void* stream) {
  using namespace davet;
  using namespace davet::unm;
  if (batch < 0 || total_rows < 0 || V < 8 || V % 8 != 0 || k < 1 || k > 1024) return DAVET_ERR_INVALID_ARG;
  if (batch == 0) return DAVET_OK;
  if (!cu_resp_dev || !masked_dev || !tokens_dev) return DAVET_ERR_INVALID_ARG;
  if (total_rows > 0 && !logits) return DAVET_ERR_INVALID_ARG;
  if (reinterpret_cast<uintptr_t>(logits) & 15u) return DAVET_ERR_INVALID_ARG;
  if (batch > 65535 || total_rows > (int64_t(1) << 31) / 64) return DAVET_ERR_UNSUPPORTED;
  const Layout L = layout_for(total_rows, V, kNoAllocScratchBytes);
  if (L.bytes > kNoAllocScratchBytes) return DAVET_ERR_UNSUPPORTED;  // too many answer rows for the array
  davet_status st = DAVET_OK;
  uint8_t* ws = noalloc_scratch(&st);
  if (!ws) return st;
  return enqueue(logits, V, cu_resp_dev, batch, total_rows, k, masked_dev, tokens_dev, argmax_dev, conf_dev,
                 committed_dev, stats_dev, ws, L, static_cast<cudaStream_t>(stream));
}
