// unmask.cu -- confidence-ranked commitment of one denoising step (Sec. 3.1,
// Eq. 1-2) and the step statistics that feed the trajectory risk (Eq. 7).
//
// Two kernels:
//  1. row pass: each (masked row, vocabulary split) is one block that streams
//     its slice of bf16 logits once with 128-bit loads and keeps, per thread,
//     an online (max, sum of 2^(x*log2e - max*log2e), first argmax) triple;
//     triples merge with warp shuffles and shared memory into one partial per
//     (row, split) in the workspace.
//  2. select: one block per request merges the splits of its masked rows
//     into (argmax, conf = 1/sum), counts churn against the previous argmax,
//     then takes the top-k rows by (conf desc, position asc) with k rounds
//     of a block-wide arg-max and commits them.
#include <algorithm>
#include <climits>
#include <mutex>

#include "common.cuh"

namespace davet {
namespace unm {

constexpr int kRowThreads = 256;
constexpr int kSelThreads = 256;
constexpr float kLog2e = 1.4426950408889634f;

struct Partial {
  float m;    // max logit * log2(e)
  float s;    // sum of 2^(x*log2e - m)
  int idx;    // first index attaining the max
  int pad;
};

struct Layout {
  int nsplit;
  size_t off_partial, off_conf, off_idx, bytes;
};

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

inline Layout layout_for(int64_t total_rows, int V, int batch = 0) {
  Layout L;
  const int64_t v8 = V / 8;
  // about six waves of 8 blocks per SM when every row is masked, so the grid
  // keeps a short tail as rows are committed; each split keeps at least 1024
  // 16-byte slices (16 KB) so the block-level merge stays cheap
  int64_t want = total_rows > 0 ? (152 * 8 * 6 + total_rows - 1) / total_rows : 1;
  const int64_t cap = std::max<int64_t>(1, v8 / 1024);
  L.nsplit = static_cast<int>(std::max<int64_t>(1, std::min<int64_t>(std::min<int64_t>(want, cap), 64)));
  L.off_partial = 0;
  L.off_conf = align256(static_cast<size_t>(total_rows) * L.nsplit * sizeof(Partial));
  L.off_idx = L.off_conf + align256(static_cast<size_t>(total_rows) * sizeof(float));
  L.bytes = L.off_idx + align256(static_cast<size_t>(total_rows) * sizeof(int));
  (void)batch;
  return L;
}

__device__ __forceinline__ Partial merge(Partial a, Partial b) {
  Partial r;
  r.m = fmaxf(a.m, b.m);
  const float sa = a.s > 0.f ? a.s * ex2(a.m - r.m) : 0.f;
  const float sb = b.s > 0.f ? b.s * ex2(b.m - r.m) : 0.f;
  r.s = sa + sb;
  r.idx = a.m > b.m ? a.idx : (b.m > a.m ? b.idx : min(a.idx, b.idx));
  r.pad = 0;
  return r;
}

__device__ __forceinline__ Partial shfl_merge(Partial p) {
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    Partial q;
    q.m = __shfl_xor_sync(0xffffffffu, p.m, o);
    q.s = __shfl_xor_sync(0xffffffffu, p.s, o);
    q.idx = __shfl_xor_sync(0xffffffffu, p.idx, o);
    p = merge(p, q);
  }
  return p;
}

__device__ __forceinline__ uint4 ld_stream(const uint4* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

// Fold one 16-byte slice (8 logits starting at vocabulary index w0) into p.
__device__ __forceinline__ void fold(Partial& p, uint4 u, int w0) {
  float x[8];
  x[0] = bf16lo(u.x) * kLog2e; x[1] = bf16hi(u.x) * kLog2e;
  x[2] = bf16lo(u.y) * kLog2e; x[3] = bf16hi(u.y) * kLog2e;
  x[4] = bf16lo(u.z) * kLog2e; x[5] = bf16hi(u.z) * kLog2e;
  x[6] = bf16lo(u.w) * kLog2e; x[7] = bf16hi(u.w) * kLog2e;
  float vm = x[0];
#pragma unroll
  for (int k = 1; k < 8; ++k) vm = fmaxf(vm, x[k]);
  if (vm > p.m) {
    int first = 7;
#pragma unroll
    for (int k = 6; k >= 0; --k) first = (x[k] == vm) ? k : first;
    p.idx = w0 + first;
    p.s = p.s > 0.f ? p.s * ex2(p.m - vm) : 0.f;
    p.m = vm;
  }
  // pairwise sum of the eight terms, then one add into the running sum
  float e[8];
#pragma unroll
  for (int k = 0; k < 8; ++k) e[k] = ex2(x[k] - p.m);
  p.s += ((e[0] + e[1]) + (e[2] + e[3])) + ((e[4] + e[5]) + (e[6] + e[7]));
}

__global__ void __launch_bounds__(kRowThreads) row_pass(const uint4* __restrict__ logits, int V8,
                                                        const uint8_t* __restrict__ masked, long long total_rows,
                                                        int nsplit, Partial* __restrict__ out) {
  pdl_launch_dependents();
  pdl_wait();
  const long long item = blockIdx.x;
  const long long row = item / nsplit;
  const int split = static_cast<int>(item - row * nsplit);
  if (row >= total_rows || !masked[row]) return;
  const int per = (V8 + nsplit - 1) / nsplit;
  const int lo = split * per, hi = min(V8, lo + per);
  const uint4* base = logits + row * static_cast<long long>(V8);
  Partial p;
  p.m = -INFINITY;
  p.s = 0.f;
  p.idx = INT_MAX;
  p.pad = 0;
  int v = lo + threadIdx.x;
  for (; v + 3 * kRowThreads < hi; v += 4 * kRowThreads) {
    uint4 u[4];
#pragma unroll
    for (int k = 0; k < 4; ++k) u[k] = ld_stream(base + v + k * kRowThreads);
#pragma unroll
    for (int k = 0; k < 4; ++k) fold(p, u[k], (v + k * kRowThreads) * 8);
  }
  for (; v < hi; v += kRowThreads) fold(p, ld_stream(base + v), v * 8);

  // block merge: warps, then warp 0 over the warp results
  __shared__ Partial s_p[kRowThreads / 32];
  p = shfl_merge(p);
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  if (lane == 0) s_p[warp] = p;
  __syncthreads();
  if (warp == 0) {
    Partial q;
    if (lane < kRowThreads / 32) {
      q = s_p[lane];
    } else {
      q.m = -INFINITY; q.s = 0.f; q.idx = INT_MAX; q.pad = 0;
    }
    q = shfl_merge(q);
    if (lane == 0) out[item] = q;
  }
}

struct SelArgs {
  const Partial* partial;
  int nsplit;
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
  float* row_conf;  // workspace: conf of masked rows
  int32_t* row_idx; // workspace: argmax of masked rows
  unsigned* err;
};

// Block-wide arg-max of (conf, -pos): returns the winning row (or -1).
__device__ __forceinline__ long long block_best(float c, long long pos, float* s_c, long long* s_pos) {
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
  for (int o = 16; o > 0; o >>= 1) {
    const float c2 = __shfl_xor_sync(0xffffffffu, c, o);
    const long long p2 = __shfl_xor_sync(0xffffffffu, pos, o);
    if (c2 > c || (c2 == c && p2 < pos)) { c = c2; pos = p2; }
  }
  if (lane == 0) { s_c[warp] = c; s_pos[warp] = pos; }
  __syncthreads();
  if (warp == 0) {
    c = lane < kSelThreads / 32 ? s_c[lane] : -2.f;
    pos = lane < kSelThreads / 32 ? s_pos[lane] : LLONG_MAX;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
      const float c2 = __shfl_xor_sync(0xffffffffu, c, o);
      const long long p2 = __shfl_xor_sync(0xffffffffu, pos, o);
      if (c2 > c || (c2 == c && p2 < pos)) { c = c2; pos = p2; }
    }
    if (lane == 0) { s_c[0] = c; s_pos[0] = pos; }
  }
  __syncthreads();
  const long long best = (s_c[0] >= 0.f) ? s_pos[0] : -1;
  __syncthreads();
  return best;
}

// Merge the splits of request b's masked rows, count churn, take the top-k
// and commit; run by one block of kSelThreads threads.
__device__ __forceinline__ void select_request(const SelArgs& a, int b) {
  const long long cu0 = a.cu[b], cu1 = a.cu[b + 1];
  const long long s0 = min(max(cu0, 0LL), a.total_rows);
  const long long s1 = min(max(cu1, s0), a.total_rows);
  if (threadIdx.x == 0 && (cu0 != s0 || cu1 != s1)) raise_error(a.err, DEV_ERR_ARG);

  __shared__ float s_c[kSelThreads / 32];
  __shared__ long long s_pos[kSelThreads / 32];
  __shared__ float s_sum[kSelThreads / 32];
  __shared__ int s_cnt[3][kSelThreads / 32];

  float conf_sum = 0.f;
  int n_masked = 0, n_both = 0, n_changed = 0;
  for (long long i = s0 + threadIdx.x; i < s1; i += kSelThreads) {
    if (!a.masked[i]) continue;
    // load the row's partials eight at a time, then merge them
    Partial p = a.partial[i * a.nsplit];
    for (int sp0 = 1; sp0 < a.nsplit; sp0 += 8) {
      Partial q[8];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (sp0 + u < a.nsplit) q[u] = a.partial[i * a.nsplit + sp0 + u];
#pragma unroll
      for (int u = 0; u < 8; ++u)
        if (sp0 + u < a.nsplit) p = merge(p, q[u]);
    }
    const int idx = p.idx == INT_MAX ? 0 : p.idx;
    const float conf = 1.f / p.s;
    a.row_conf[i] = conf;
    a.row_idx[i] = idx;
    if (a.conf_out) a.conf_out[i] = conf;
    if (a.argmax) {
      const int prev = a.argmax[i];
      if (prev >= 0) {
        ++n_both;
        n_changed += prev != idx;
      }
      a.argmax[i] = idx;
    }
    conf_sum += conf;
    ++n_masked;
  }
  // block sums (fixed order: per warp, then warps in order)
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
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
  float tot_conf = 0.f;
  int tot_masked = 0, tot_both = 0, tot_changed = 0;
  for (int w = 0; w < kSelThreads / 32; ++w) {
    tot_conf += s_sum[w];
    tot_masked += s_cnt[0][w];
    tot_both += s_cnt[1][w];
    tot_changed += s_cnt[2][w];
  }
  if (threadIdx.x == 0 && a.stats) {
    a.stats[2 * b + 0] = tot_masked ? tot_conf / static_cast<float>(tot_masked) : 0.f;
    a.stats[2 * b + 1] = tot_both ? static_cast<float>(tot_changed) / static_cast<float>(tot_both) : 0.f;
  }

  // top-k: k rounds of a block-wide arg-max over the rows still masked
  const int take = min(a.k, tot_masked);
  for (int j = 0; j < take; ++j) {
    float best_c = -2.f;
    long long best_pos = LLONG_MAX;
    for (long long i = s0 + threadIdx.x; i < s1; i += kSelThreads) {
      if (!a.masked[i]) continue;
      const float c = a.row_conf[i];
      if (c > best_c || (c == best_c && i < best_pos)) { best_c = c; best_pos = i; }
    }
    const long long w = block_best(best_c, best_pos, s_c, s_pos);
    if (threadIdx.x == 0 && w >= 0) {
      a.tokens[w] = a.row_idx[w];
      a.masked[w] = 0;
      if (a.committed) a.committed[static_cast<long long>(b) * a.k + j] = static_cast<int32_t>(w - s0);
    }
    __syncthreads();
  }
  if (a.committed)
    for (int j = take + threadIdx.x; j < a.k; j += kSelThreads) a.committed[static_cast<long long>(b) * a.k + j] = -1;
}


__global__ void __launch_bounds__(kSelThreads) select_commit(SelArgs a) {
  pdl_launch_dependents();
  pdl_wait();
  select_request(a, blockIdx.x);
}

}  // namespace unm
}  // namespace davet

extern "C" davet_status davet_unmask_topk_workspace(int64_t total_rows, int V, int batch, size_t* bytes) {
  if (total_rows < 0 || V < 8 || V % 8 != 0 || batch < 0 || !bytes) return DAVET_ERR_INVALID_ARG;
  *bytes = davet::unm::layout_for(total_rows, V, batch).bytes;
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
  const Layout L = layout_for(total_rows, V, batch);
  if (workspace_bytes < L.bytes) return DAVET_ERR_INVALID_ARG;
  unsigned* err = device_error_word();
  if (!err) return DAVET_ERR_CUDA;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  Partial* partial = reinterpret_cast<Partial*>(ws + L.off_partial);
  SelArgs a;
  a.partial = partial;
  a.nsplit = L.nsplit;
  a.cu = cu_resp_dev;
  a.batch = batch;
  a.total_rows = total_rows;
  a.k = k;
  a.masked = masked_dev;
  a.tokens = tokens_dev;
  a.argmax = argmax_dev;
  a.conf_out = conf_dev;
  a.committed = committed_dev;
  a.stats = stats_dev;
  a.row_conf = reinterpret_cast<float*>(ws + L.off_conf);
  a.row_idx = reinterpret_cast<int32_t*>(ws + L.off_idx);
  a.err = err;
  if (total_rows > 0) {
    const long long items = total_rows * L.nsplit;
    const cudaError_t e = launch(row_pass, dim3(static_cast<unsigned>(items)), dim3(kRowThreads), 0, st,
                                 static_cast<const uint4*>(logits), V / 8, static_cast<const uint8_t*>(masked_dev),
                                 static_cast<long long>(total_rows), L.nsplit, partial);
    if (e != cudaSuccess) return cuda_fail(e);
  }
  const cudaError_t e = launch(select_commit, dim3(batch), dim3(kSelThreads), 0, st, a);
  return e == cudaSuccess ? DAVET_OK : cuda_fail(e);
}

// ---------------------------------------------------------------------------
// Allocation-free variant of davet_unmask_topk.
//
// Its scratch lives in a fixed device array owned by the library, so the
// caller passes only inputs and outputs.  Every device that loads the library
// keeps this array for the life of the process, and all calls on a device
// share it.
namespace davet {
namespace unm {

constexpr size_t kNoAllocScratchBytes = size_t(1) << 20;  // DAVET_NOALLOC_SCRATCH_BYTES
static __device__ __align__(256) unsigned char g_noalloc_scratch[kNoAllocScratchBytes];

constexpr int kNoAllocMaxDevices = 64;
static uint8_t* g_noalloc_addr[kNoAllocMaxDevices] = {};
static std::mutex g_noalloc_mu;

// Device address of g_noalloc_scratch on the current device.  Host code only
// sees a host-side stand-in for the array under its name, so the address is
// asked for once per device, with that device current, and cached.
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
  if (!g_noalloc_addr[dev]) {
    void* p = nullptr;
    e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) {
      *st = cuda_fail(e);
      return nullptr;
    }
    g_noalloc_addr[dev] = static_cast<uint8_t*>(p);
  }
  return g_noalloc_addr[dev];
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
  const Layout L = layout_for(total_rows, V);
  if (L.bytes > kNoAllocScratchBytes) return DAVET_ERR_UNSUPPORTED;  // too many answer rows for the array
  davet_status st = DAVET_OK;
  uint8_t* ws = noalloc_scratch(&st);
  if (!ws) return st;
  unsigned* err = device_error_word();
  if (!err) return DAVET_ERR_CUDA;
  cudaStream_t s = static_cast<cudaStream_t>(stream);
  // Nothing in the scratch needs clearing: the select kernel reads only the
  // partials, confidences and argmaxes of masked rows, and the row pass of
  // this same call writes all of them first.
  Partial* partial = reinterpret_cast<Partial*>(ws + L.off_partial);
  if (total_rows > 0) {
    const long long items = total_rows * L.nsplit;
    row_pass<<<static_cast<unsigned>(items), kRowThreads, 0, s>>>(static_cast<const uint4*>(logits), V / 8,
                                                                  masked_dev, total_rows, L.nsplit, partial);
    const davet_status e = check_launch();
    if (e != DAVET_OK) return e;
  }
  SelArgs a;
  a.partial = partial;
  a.nsplit = L.nsplit;
  a.cu = cu_resp_dev;
  a.batch = batch;
  a.total_rows = total_rows;
  a.k = k;
  a.masked = masked_dev;
  a.tokens = tokens_dev;
  a.argmax = argmax_dev;
  a.conf_out = conf_dev;
  a.committed = committed_dev;
  a.stats = stats_dev;
  a.row_conf = reinterpret_cast<float*>(ws + L.off_conf);
  a.row_idx = reinterpret_cast<int32_t*>(ws + L.off_idx);
  a.err = err;
  select_commit<<<batch, kSelThreads, 0, s>>>(a);
  return check_launch();
}
