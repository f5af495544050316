// gemm.cu -- the dense projections of a full transformer layer (QKV, output,
// gated MLP, LM head) as one tcgen05 GEMM with fused epilogues:
//   out[M, N'] = epilogue(A[M, K] . W[N, K]^T)
// A and W are row-major bf16 with K contiguous (W as a linear layer's weight).
//
// Persistent, warp-specialized, one CTA per SM, 192 threads:
//   warp 0     TMA producer: 128 x 64 tiles of A and 256 x 64 tiles of W
//              (128-byte swizzle) into a 4-stage ring;
//   warp 1     owns TMEM (512 columns: two 128 x 256 fp32 accumulators) and
//              issues the MMAs (one thread, M = 128, N = 256, K = 16 each);
//   warps 2-5  epilogue: thread r of the four warps owns accumulator row r,
//              reads it from TMEM 32 columns at a time, applies the epilogue
//              and writes bf16 into the warp's two 32 x 64 shared-memory
//              slabs (128-byte swizzle), which the warp's lane 0 stores with
//              TMA (full 128-byte lines; the threads do not wait for the
//              writes); it runs on one accumulator while the MMAs fill the
//              other.  A warp whose 32 rows are not all below M stores its
//              valid rows directly instead.
// Output tiles are visited m-fastest, so the CTAs working at the same time
// share one 256-row block of W through L2.
// Epilogues: plain store; residual add (out = residual + product, in place
// allowed); gated MLP (W holds gate and up rows interleaved in blocks of
// 128: columns [0,128) of each tile are the gate, [128,256) the up
// projection; out = silu(gate) * up, half as many columns); rotary position
// embedding on the query and key columns (pairs (d, d + D/2) of each head,
// angle from a cos/sin table indexed by the row's position in its request;
// the table is frequency-major, so the lanes of a warp, rows at consecutive
// positions, read consecutive entries).
// Around every epilogue: an optional row scale 1/rms from partial sums of
// squares (an RMS normalization of A folded into the product, its gain in W)
// and, for the store and residual epilogues, the sums of squares of the
// stored rows per 256 columns (the next product's normalization input).
// M > 128 runs on CTA pairs (gemm2_kernel below), with a K split into fp32
// partials and a reduction kernel when the tiles leave most pairs idle.
// A row count on the device (rows_dev) limits every kernel to the rows the
// step has; each kernel keeps it in a scalar of its own.
#include <algorithm>
#include <mutex>

#include "common.cuh"

namespace davet {
namespace gemm {

constexpr int BM = 128, BN = 256, BK = 64, STAGES = 4;
constexpr int kThreads = 192;
constexpr int kWarpTma = 0, kWarpMma = 1;  // warps 2-5: epilogue
constexpr int kTmemCols = 512;
constexpr uint32_t kStageA = BM * BK * 2;  // 16 KB
constexpr uint32_t kStageB = BN * BK * 2;  // 32 KB

enum : int { EPI_STORE = 0, EPI_RESIDUAL = 1, EPI_SWIGLU = 2, EPI_ROPE = 3 };

constexpr uint32_t kSlab = 32 * 128;  // an epilogue warp's 32 rows x 64 bf16 columns: 4 KB

struct Smem {
  alignas(1024) uint8_t a[STAGES][kStageA];
  alignas(1024) uint8_t b[STAGES][kStageB];
  alignas(1024) uint8_t epi[4][2][kSlab];  // [epilogue warp][slab]
  uint64_t full[STAGES], empty[STAGES];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t fin;
  uint32_t tmem;
  int abort;
};

struct Params {
  long long M;
  int N, K;
  int tiles_m, tiles_n;
  uint16_t* out;
  int ldo;  // output row stride (elements)
  const uint16_t* residual;
  int epi;
  // rotary embedding
  const int32_t* cu;  // int32 [batch + 1] request row boundaries
  int batch;
  int rope_cols;  // columns [0, rope_cols) are query and key heads
  int head_dim;
  int max_pos;
  const float2* rope;  // [head_dim / 2][max_pos] (cos, sin), frequency-major
  unsigned* err;
  // split of K (CTA-pair kernel): `split` slices of `kb_per` k-blocks (the last
  // takes the rest) write fp32 partials [split][tiles_n][M rounded to 256][256]
  int split;
  int kb_per;
  float* part;
  // nullable: the row count on the device (at most M), read after the
  // previous kernel finished; rows from there on are neither computed nor stored
  const int32_t* rows_dev;
  // normalization folded into the product (nullable): row r of the product
  // is scaled by 1 / sqrt(sum_j rss[r * rss_parts + j] / K + rss_eps) before
  // the epilogue, i.e. A's rows are RMS-normalized (the gain is in W)
  const float* rss;
  int rss_parts;
  float rss_eps;
  // nullable (store and residual epilogues): ss_out[r * tiles_n + n-block] =
  // sum of squares of the row's 256 stored bf16 values, for the next
  // product's normalization
  float* ss_out;
};

// 1 / rms of A's row from its partial sums of squares (1 without them).
__device__ __forceinline__ float row_scale(const Params& p, long long row, bool row_ok) {
  if (!p.rss || !row_ok) return 1.0f;
  const float* s = p.rss + row * p.rss_parts;
  float t = 0.0f;
  for (int j = 0; j < p.rss_parts; ++j) t += s[j];
  return rsqrtf(t / static_cast<float>(p.K) + p.rss_eps);
}

// A device row count clamped to [0, M]; a count outside that range sets a
// bit of the device error word (capacity above M, argument below 0), raised
// by one thread per block.
__device__ __forceinline__ long long clamp_rows(const int32_t* rows_dev, long long M, unsigned* err) {
  const long long m = *rows_dev;
  if ((m < 0 || m > M) && threadIdx.x == 0) raise_error(err, m < 0 ? DEV_ERR_ARG : DEV_ERR_CAPACITY);
  return m < 0 ? 0 : (m < M ? m : M);
}

// The launch's row count: M, or the smaller count on the device.  Kernels
// keep it in a scalar of their own rather than in their copy of the
// parameters.
__device__ __forceinline__ long long rows_now(const Params& p) {
  if (!p.rows_dev) return p.M;
  return clamp_rows(p.rows_dev, p.M, p.err);
}

__device__ __forceinline__ void tma_load_2d(void* dst, const void* tmap, uint64_t* bar, int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(smem_u32(bar)), "r"(c0), "r"(c1)
      : "memory");
}

__device__ __forceinline__ bool warp_wait(uint64_t* bar, uint32_t parity, unsigned* err, volatile int* abort_flag) {
  const bool ok = mbar_wait(bar, parity, err, abort_flag);
  return __all_sync(0xffffffffu, ok);
}

// silu(g) = g * sigmoid(g); the fast division is exact enough for a bf16 output
__device__ __forceinline__ float silu(float g) { return __fdividef(g, 1.0f + __expf(-g)); }

// sum of squares of the 8 bf16 values of a 16-byte word
__device__ __forceinline__ float sumsq8(uint4 w) {
  float s = 0.0f;
  s = fmaf(bf16lo(w.x), bf16lo(w.x), s); s = fmaf(bf16hi(w.x), bf16hi(w.x), s);
  s = fmaf(bf16lo(w.y), bf16lo(w.y), s); s = fmaf(bf16hi(w.y), bf16hi(w.y), s);
  s = fmaf(bf16lo(w.z), bf16lo(w.z), s); s = fmaf(bf16hi(w.z), bf16hi(w.z), s);
  s = fmaf(bf16lo(w.w), bf16lo(w.w), s); s = fmaf(bf16hi(w.w), bf16hi(w.w), s);
  return s;
}

// Stores 32 values as bf16; returns the sum of squares of the stored values.
__device__ __forceinline__ float store32(uint16_t* dst, const float (&v)[32]) {
  uint4* d4 = reinterpret_cast<uint4*>(dst);
  float ss = 0.0f;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    uint4 w;
    w.x = pack_bf16x2(v[8 * u + 0], v[8 * u + 1]);
    w.y = pack_bf16x2(v[8 * u + 2], v[8 * u + 3]);
    w.z = pack_bf16x2(v[8 * u + 4], v[8 * u + 5]);
    w.w = pack_bf16x2(v[8 * u + 6], v[8 * u + 7]);
    d4[u] = w;
    ss += sumsq8(w);
  }
  return ss;
}

__device__ __forceinline__ void load_acc32(uint32_t taddr, float (&v)[32]) {
  uint32_t r[32];
  tmem_ld32(taddr, r);
  tmem_wait_ld();
#pragma unroll
  for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// The epilogue of one output row of a 256-column tile: `get(c, v)` fills
// v[0..32) with the fp32 products of columns [c, c + 32) of the row (a
// warp-collective TMEM load: every lane calls it), and the row's stores
// happen only where row_ok.
template <class Get>
__device__ __forceinline__ void epilogue_row(const Params& p, long long row, bool row_ok, int n0, Get&& get) {
  if (p.epi == EPI_SWIGLU) {
    uint16_t* dst = p.out + row * p.ldo + n0 / 2;
#pragma unroll 1
    for (int c = 0; c < BN / 2; c += 32) {
      float g[32], u[32];
      get(c, g);
      get(BN / 2 + c, u);
#pragma unroll
      for (int i = 0; i < 32; ++i) g[i] = silu(g[i]) * u[i];
      if (row_ok) store32(dst + c, g);
    }
  } else if (p.epi == EPI_ROPE && n0 < p.rope_cols) {
    // the row's position in its request
    int pos = 0;
    if (row_ok) {
      int lo = 0, hi = p.batch;  // largest b with cu[b] <= row
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (p.cu[mid] <= row) lo = mid; else hi = mid;
      }
      pos = static_cast<int>(row - p.cu[lo]);
      if (pos >= p.max_pos) {
        raise_error(p.err, DEV_ERR_ARG);
        pos = p.max_pos - 1;
      }
    }
    const int half = p.head_dim / 2;
    const float2* tab = p.rope + pos;  // frequency d at tab[d * max_pos]
    uint16_t* dst = p.out + row * p.ldo + n0;
#pragma unroll 1
    for (int hb = 0; hb < BN; hb += p.head_dim) {
#pragma unroll 1
      for (int c = 0; c < half; c += 32) {
        float x[32], y[32];
        get(hb + c, x);
        get(hb + half + c, y);
        if (row_ok) {
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float2 cs = tab[static_cast<long long>(c + i) * p.max_pos];
            const float a = x[i], b = y[i];
            x[i] = a * cs.x - b * cs.y;
            y[i] = b * cs.x + a * cs.y;
          }
          store32(dst + hb + c, x);
          store32(dst + hb + half + c, y);
        }
      }
    }
  } else {
    uint16_t* dst = p.out + row * p.ldo + n0;
    const uint16_t* res = p.epi == EPI_RESIDUAL ? p.residual + row * p.ldo + n0 : nullptr;
    float ss = 0.0f;
#pragma unroll 1
    for (int c = 0; c < BN; c += 32) {
      float v[32];
      get(c, v);
      if (row_ok) {
        if (res) {
          const uint4* r4 = reinterpret_cast<const uint4*>(res + c);
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const uint4 w = r4[u];
            v[8 * u + 0] += bf16lo(w.x); v[8 * u + 1] += bf16hi(w.x);
            v[8 * u + 2] += bf16lo(w.y); v[8 * u + 3] += bf16hi(w.y);
            v[8 * u + 4] += bf16lo(w.z); v[8 * u + 5] += bf16hi(w.z);
            v[8 * u + 6] += bf16lo(w.w); v[8 * u + 7] += bf16hi(w.w);
          }
        }
        ss += store32(dst + c, v);
      }
    }
    if (p.ss_out && row_ok) p.ss_out[row * p.tiles_n + n0 / BN] = ss;
  }
}

__device__ __forceinline__ void tma_store_2d(const void* tmap, const void* src, int c0, int c1) {
  asm volatile("cp.async.bulk.tensor.2d.global.shared::cta.bulk_group [%0, {%2, %3}], [%1];" ::"l"(
                   reinterpret_cast<uint64_t>(tmap)),
               "r"(smem_u32(src)), "r"(c0), "r"(c1)
               : "memory");
}
__device__ __forceinline__ void bulk_commit() { asm volatile("cp.async.bulk.commit_group;" ::: "memory"); }
// the shared-memory sources of this thread's bulk stores have been read
__device__ __forceinline__ void bulk_wait_read() { asm volatile("cp.async.bulk.wait_group.read 0;" ::: "memory"); }
// ... and their writes are done
__device__ __forceinline__ void bulk_wait_all() { asm volatile("cp.async.bulk.wait_group 0;" ::: "memory"); }

// 32 values of this lane's row into a 32 x 64 slab, columns [col, col + 32)
// (col 0 or 32), in the 128-byte swizzle the output map uses: 16-byte chunk
// j of row r sits at r * 128 + (j ^ (r % 8)) * 16 (conflict-free per warp).
// Returns the sum of squares of the staged bf16 values.
__device__ __forceinline__ float stage32(uint8_t* slab, int lane, int col, const float (&v)[32]) {
  float ss = 0.0f;
#pragma unroll
  for (int u = 0; u < 4; ++u) {
    uint4 w;
    w.x = pack_bf16x2(v[8 * u + 0], v[8 * u + 1]);
    w.y = pack_bf16x2(v[8 * u + 2], v[8 * u + 3]);
    w.z = pack_bf16x2(v[8 * u + 4], v[8 * u + 5]);
    w.w = pack_bf16x2(v[8 * u + 6], v[8 * u + 7]);
    const int j = (col >> 3) + u;
    *reinterpret_cast<uint4*>(slab + lane * 128 + ((j ^ (lane & 7)) << 4)) = w;
    ss += sumsq8(w);
  }
  return ss;
}

// 32 fp32 values of this lane's row into a 32 x 32 fp32 slab, same swizzle.
__device__ __forceinline__ void stage32_f32(uint8_t* slab, int lane, const float (&v)[32]) {
#pragma unroll
  for (int j = 0; j < 8; ++j)
    *reinterpret_cast<float4*>(slab + lane * 128 + ((j ^ (lane & 7)) << 4)) =
        make_float4(v[4 * j], v[4 * j + 1], v[4 * j + 2], v[4 * j + 3]);
}

// The epilogue of one warp's 32 rows [row0, row0 + 32), all below M, of a
// 256-column tile at column n0, in groups of 128 output columns: the group
// goes through the warp's two slabs and out with two TMA stores of 32 x 64.
// `get` is the TMEM read of epilogue_row.
template <class Get>
__device__ __forceinline__ void epilogue_warp_staged(const Params& p, const void* tmap_out, uint8_t* slab0,
                                                     uint8_t* slab1, int lane, long long row0, int n0, Get&& get) {
  const long long row = row0 + lane;
  const bool swiglu = p.epi == EPI_SWIGLU, rope = p.epi == EPI_ROPE && n0 < p.rope_cols;
  const int out0 = swiglu ? n0 / 2 : n0;
  float ss = 0.0f;  // of the stored values (store and residual epilogues)
  int pos = 0;
  if (rope) {
    int lo = 0, hi = p.batch;  // largest b with cu[b] <= row
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (p.cu[mid] <= row) lo = mid; else hi = mid;
    }
    pos = static_cast<int>(row - p.cu[lo]);
    if (pos >= p.max_pos) {
      raise_error(p.err, DEV_ERR_ARG);
      pos = p.max_pos - 1;
    }
  }
#pragma unroll 1
  for (int g = 0; g < (swiglu ? 1 : 2); ++g) {
    if (lane == 0) bulk_wait_read();  // the previous group's stores have left the slabs
    __syncwarp();
    if (swiglu) {
#pragma unroll 1
      for (int c = 0; c < 128; c += 32) {
        float a[32], u[32];
        get(c, a);
        get(128 + c, u);
#pragma unroll
        for (int i = 0; i < 32; ++i) a[i] = silu(a[i]) * u[i];
        stage32(c < 64 ? slab0 : slab1, lane, c & 63, a);
      }
    } else if (rope) {
      const int half = p.head_dim / 2;
#pragma unroll 1
      for (int hb = 128 * g; hb < 128 * g + 128; hb += p.head_dim) {
#pragma unroll 1
        for (int c = 0; c < half; c += 32) {
          float x[32], y[32];
          get(hb + c, x);
          get(hb + half + c, y);
          const float2* tab = p.rope + static_cast<long long>(c) * p.max_pos + pos;
#pragma unroll
          for (int i = 0; i < 32; ++i) {
            const float2 cs = tab[static_cast<long long>(i) * p.max_pos];
            const float a = x[i], b = y[i];
            x[i] = a * cs.x - b * cs.y;
            y[i] = b * cs.x + a * cs.y;
          }
          const int cx = hb + c - 128 * g, cy = cx + half;
          stage32(cx < 64 ? slab0 : slab1, lane, cx & 63, x);
          stage32(cy < 64 ? slab0 : slab1, lane, cy & 63, y);
        }
      }
    } else {
      const uint16_t* res = p.epi == EPI_RESIDUAL ? p.residual + row * p.ldo + n0 + 128 * g : nullptr;
#pragma unroll 1
      for (int c = 0; c < 128; c += 32) {
        float v[32];
        get(128 * g + c, v);
        if (res) {
          const uint4* r4 = reinterpret_cast<const uint4*>(res + c);
#pragma unroll
          for (int u = 0; u < 4; ++u) {
            const uint4 w = r4[u];
            v[8 * u + 0] += bf16lo(w.x); v[8 * u + 1] += bf16hi(w.x);
            v[8 * u + 2] += bf16lo(w.y); v[8 * u + 3] += bf16hi(w.y);
            v[8 * u + 4] += bf16lo(w.z); v[8 * u + 5] += bf16hi(w.z);
            v[8 * u + 6] += bf16lo(w.w); v[8 * u + 7] += bf16hi(w.w);
          }
        }
        ss += stage32(c < 64 ? slab0 : slab1, lane, c & 63, v);
      }
    }
    fence_proxy_async_smem();  // the slabs' generic writes, visible to the TMA unit
    __syncwarp();
    if (lane == 0) {
      tma_store_2d(tmap_out, slab0, out0 + 128 * g, static_cast<int>(row0));
      tma_store_2d(tmap_out, slab1, out0 + 128 * g + 64, static_cast<int>(row0));
      bulk_commit();
    }
  }
  if (p.ss_out && !swiglu && !rope) p.ss_out[row * p.tiles_n + n0 / BN] = ss;
}

__global__ void __launch_bounds__(kThreads, 1)
    gemm_kernel(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_w,
                const __grid_constant__ CUtensorMap tmap_out, Params p0) {
  extern __shared__ uint8_t smem_raw[];
  const Params& p = p0;
  Smem& s = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  volatile int* abort_flag = &s.abort;

  if (tid == 0) {
    s.abort = 0;
    for (int i = 0; i < STAGES; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.acc_full[i], 1);
      mbar_init(&s.acc_empty[i], 4);  // one arrival per epilogue warp
    }
    mbar_init(&s.fin, 1);
    fence_mbar_init();
  }
  if (warp == kWarpMma) {
    tmem_alloc(&s.tmem, kTmemCols);
    tmem_relinquish();
  }
  if (warp == kWarpTma && lane == 0) {
    tma_prefetch_desc(&tmap_a);
    tma_prefetch_desc(&tmap_w);
    tma_prefetch_desc(&tmap_out);
  }
  pdl_launch_dependents();
  pdl_wait();  // A (and the residual) come from the previous kernel
  const long long M = rows_now(p);
  const int tiles_m = static_cast<int>((M + BM - 1) / BM);
  tc_fence_before();
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = s.tmem;
  const int n_tiles = tiles_m * p.tiles_n;
  const int nk = p.K / BK;

  if (warp == kWarpTma) {
    if (lane == 0) {
      uint32_t it = 0;
      for (int t = blockIdx.x; t < n_tiles; t += gridDim.x) {
        const int m0 = (t % tiles_m) * BM, n0 = (t / tiles_m) * BN;
        bool ok = true;
        for (int kb = 0; kb < nk; ++kb, ++it) {
          const uint32_t st = it % STAGES;
          if (it >= STAGES && !mbar_wait(&s.empty[st], ((it / STAGES) - 1) & 1, p.err, abort_flag)) {
            ok = false;
            break;
          }
          mbar_arrive_expect_tx(&s.full[st], kStageA + kStageB);
          tma_load_2d(s.a[st], &tmap_a, &s.full[st], kb * BK, m0);
          tma_load_2d(s.b[st], &tmap_w, &s.full[st], kb * BK, n0);
        }
        if (!ok) break;
      }
    }
  } else if (warp == kWarpMma) {
    if (lane == 0) {
      constexpr uint32_t kIdesc = idesc_bf16_f32(BM, BN, false, false);
      uint32_t it = 0, tc = 0;
      bool ok = true;
      for (int t = blockIdx.x; ok && t < n_tiles; t += gridDim.x, ++tc) {
        const uint32_t ab = tc & 1, use = tc >> 1;
        if (use > 0 && !mbar_wait(&s.acc_empty[ab], (use - 1) & 1, p.err, abort_flag)) break;
        tc_fence_after();
        const uint32_t d = tmem + ab * BN;
        for (int kb = 0; kb < nk; ++kb, ++it) {
          const uint32_t st = it % STAGES;
          if (!mbar_wait(&s.full[st], (it / STAGES) & 1, p.err, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t da = sw128_desc(smem_u32(s.a[st]), 16, 1024);
          const uint64_t db = sw128_desc(smem_u32(s.b[st]), 16, 1024);
          if (kb == 0)
            umma_ss_imm<false>(d, da, db, kIdesc);
          else
            umma_ss_imm<true>(d, da, db, kIdesc);
          umma_ss_imm<true>(d, da + 2, db + 2, kIdesc);
          umma_ss_imm<true>(d, da + 4, db + 4, kIdesc);
          umma_ss_imm<true>(d, da + 6, db + 6, kIdesc);
          umma_commit(&s.empty[st]);
        }
        if (ok) umma_commit(&s.acc_full[ab]);
      }
      // every issued MMA completes before TMEM is released
      umma_commit(&s.fin);
      mbar_wait(&s.fin, 0, p.err, nullptr);
    }
  } else {
    // ------------------------------------------------------------ epilogue
    const int q = warp & 3;  // TMEM lane quarter this warp may access
    const int r = 32 * q + lane;
    uint32_t tc = 0;
    for (int t = blockIdx.x; t < n_tiles; t += gridDim.x, ++tc) {
      const uint32_t ab = tc & 1, use = tc >> 1;
      if (!warp_wait(&s.acc_full[ab], use & 1, p.err, abort_flag)) break;
      tc_fence_after();
      const int m0 = (t % tiles_m) * BM, n0 = (t / tiles_m) * BN;
      const long long row = static_cast<long long>(m0) + r;
      const bool row_ok = row < M;
      const uint32_t acc = tmem + (static_cast<uint32_t>(32 * q) << 16) + ab * BN;
      const float rs = row_scale(p, row, row_ok);
      auto get = [&](int c, float (&v)[32]) {
        load_acc32(acc + c, v);
        if (p.rss) {
#pragma unroll
          for (int i = 0; i < 32; ++i) v[i] *= rs;
        }
      };
      const long long row0 = static_cast<long long>(m0) + 32 * q;
      if (row0 + 32 <= M)
        epilogue_warp_staged(p, &tmap_out, s.epi[q][0], s.epi[q][1], lane, row0, n0, get);
      else
        epilogue_row(p, row, row_ok, n0, get);
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&s.acc_empty[ab]);
    }
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  if (warp == kWarpMma) {
    tc_fence_after();
    tmem_dealloc(tmem, kTmemCols);
  }
}

// ------------------------------------------------------------ 2-SM tiles
// A cluster of two CTAs (a CTA pair on two SMs) computes a 256 x 256 tile
// with tcgen05 MMAs of M = 256 issued by the even CTA: each CTA holds its
// 128 rows of A and 128 of the tile's 256 rows of W, so each SM takes in half
// the operand bytes per FLOP of the one-CTA tile.  Each CTA's TMEM holds the
// accumulator of its 128 output rows; both CTAs run the epilogue on their own
// rows, on one of two accumulators while the MMAs fill the other.  Both
// producers' TMA copies complete on the even CTA's barrier; the MMA commits
// arrive on both CTAs' barriers; the odd CTA's epilogue signals the even
// CTA's accumulator barrier remotely.  The pair's TMEM allocation is
// collective (both CTAs get the same columns); the kernel checks it.
constexpr int ST2 = 6;
constexpr uint32_t kStageB2 = BM * BK * 2;  // 128 rows of W: 16 KB
constexpr uint32_t kTmemCols2 = 512;        // two 128 x 256 accumulators per CTA

struct Smem2 {
  alignas(1024) uint8_t a[ST2][kStageA];
  alignas(1024) uint8_t b[ST2][kStageB2];
  alignas(1024) uint8_t epi[4][2][kSlab];  // [epilogue warp][slab]
  uint64_t full[ST2], empty[ST2];
  uint64_t acc_full[2], acc_empty[2];
  uint64_t fin;
  uint32_t tmem;
  int abort;
};

__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
// Address of the same shared-memory variable in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t map_to_rank(const void* p, uint32_t rank) {
  uint32_t r;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(smem_u32(p)), "r"(rank));
  return r;
}
__device__ __forceinline__ void cluster_sync_all() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ void remote_arrive(uint32_t cluster_addr) {
  asm volatile("mbarrier.arrive.release.cluster.shared::cluster.b64 _, [%0];" ::"r"(cluster_addr) : "memory");
}
__device__ __forceinline__ void tma_load_2d_pair(void* dst, const void* tmap, uint32_t bar_cluster, int c0, int c1) {
  asm volatile(
      "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.mbarrier::complete_tx::bytes"
      " [%0], [%1, {%3, %4}], [%2];" ::"r"(smem_u32(dst)),
      "l"(reinterpret_cast<uint64_t>(tmap)), "r"(bar_cluster), "r"(c0), "r"(c1)
      : "memory");
}
template <bool ACC>
__device__ __forceinline__ void umma_pair(uint32_t d_tmem, uint64_t a_desc, uint64_t b_desc, uint32_t idesc) {
  if constexpr (ACC)
    asm volatile("tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, 1;" ::"r"(d_tmem), "l"(a_desc), "l"(b_desc),
                 "r"(idesc)
                 : "memory");
  else
    asm volatile("tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, 0;" ::"r"(d_tmem), "l"(a_desc), "l"(b_desc),
                 "r"(idesc)
                 : "memory");
}
__device__ __forceinline__ void umma_commit_pair(uint64_t* bar) {
  asm volatile(
      "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64 [%0], %1;" ::"r"(
          smem_u32(bar)),
      "h"(static_cast<uint16_t>(3))
      : "memory");
}

__global__ void __launch_bounds__(kThreads, 1)
    gemm2_kernel(const __grid_constant__ CUtensorMap tmap_a, const __grid_constant__ CUtensorMap tmap_w,
                 const __grid_constant__ CUtensorMap tmap_out, const __grid_constant__ CUtensorMap tmap_part,
                 Params p0) {
  extern __shared__ uint8_t smem_raw[];
  const Params& p = p0;
  Smem2& s = *reinterpret_cast<Smem2*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
  volatile int* abort_flag = &s.abort;
  const uint32_t rank = cluster_rank();
  const int pair = blockIdx.x >> 1, n_pairs = gridDim.x >> 1;

  if (tid == 0) {
    s.abort = 0;
    for (int i = 0; i < ST2; ++i) {
      mbar_init(&s.full[i], 1);
      mbar_init(&s.empty[i], 1);
    }
    for (int i = 0; i < 2; ++i) {
      mbar_init(&s.acc_full[i], 1);
      mbar_init(&s.acc_empty[i], 8);  // four epilogue warps in each CTA of the pair
    }
    mbar_init(&s.fin, 1);
    fence_mbar_init();
  }
  if (warp == kWarpMma) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(&s.tmem)),
                 "r"(kTmemCols2)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
  }
  if (warp == kWarpTma && lane == 0) {
    tma_prefetch_desc(&tmap_a);
    tma_prefetch_desc(&tmap_w);
    tma_prefetch_desc(&tmap_out);
    if (p.split > 1) tma_prefetch_desc(&tmap_part);
  }
  pdl_launch_dependents();
  pdl_wait();
  const long long M = rows_now(p);  // both CTAs of the pair read the same count
  tc_fence_before();
  cluster_sync_all();  // barriers initialized and TMEM allocated in both CTAs
  tc_fence_after();
  const uint32_t tmem = s.tmem;
  if (tid == 0) {
    // both CTAs must hold the accumulator at the same TMEM address
    uint32_t lead;
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(lead) : "r"(map_to_rank(&s.tmem, 0)) : "memory");
    if (lead != tmem) {
      raise_error(p.err, DEV_ERR_ARG);
      s.abort = 1;
    }
  }
  __syncthreads();
  const int tiles_m2 = static_cast<int>((M + 2 * BM - 1) / (2 * BM));
  const int n_tiles = tiles_m2 * p.tiles_n * p.split;
  const int nk = p.K / BK;
  // unit t: slice t % split of output tile t / split (m-block fastest)
  auto k_range = [&](int t, int& kb0, int& kb1) {
    const int sl = t % p.split;
    kb0 = sl * p.kb_per;
    kb1 = sl + 1 == p.split ? nk : kb0 + p.kb_per;
  };

  if (warp == kWarpTma) {
    if (lane == 0 && !s.abort) {
      uint32_t it = 0;
      bool ok = true;
      for (int t = pair; ok && t < n_tiles; t += n_pairs) {
        const int bt = t / p.split;
        const int m0 = (bt % tiles_m2) * 2 * BM + rank * BM, n0 = (bt / tiles_m2) * BN + rank * BM;
        int kb0, kb1;
        k_range(t, kb0, kb1);
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const uint32_t st = it % ST2;
          if (it >= ST2 && !mbar_wait(&s.empty[st], ((it / ST2) - 1) & 1, p.err, abort_flag)) {
            ok = false;
            break;
          }
          if (rank == 0) mbar_arrive_expect_tx(&s.full[st], 2 * (kStageA + kStageB2));
          const uint32_t bar = map_to_rank(&s.full[st], 0);
          tma_load_2d_pair(s.a[st], &tmap_a, bar, kb * BK, m0);
          tma_load_2d_pair(s.b[st], &tmap_w, bar, kb * BK, n0);
        }
      }
    }
  } else if (warp == kWarpMma) {
    if (lane == 0 && rank == 0 && !s.abort) {
      constexpr uint32_t kIdesc = idesc_bf16_f32(2 * BM, BN, false, false);
      uint32_t it = 0, tc = 0;
      bool ok = true;
      for (int t = pair; ok && t < n_tiles; t += n_pairs, ++tc) {
        const uint32_t ab = tc & 1, use = tc >> 1;
        if (use > 0 && !mbar_wait(&s.acc_empty[ab], (use - 1) & 1, p.err, abort_flag)) break;
        tc_fence_after();
        const uint32_t d = tmem + ab * BN;
        int kb0, kb1;
        k_range(t, kb0, kb1);
        for (int kb = kb0; kb < kb1; ++kb, ++it) {
          const uint32_t st = it % ST2;
          if (!mbar_wait(&s.full[st], (it / ST2) & 1, p.err, abort_flag)) {
            ok = false;
            break;
          }
          tc_fence_after();
          const uint64_t da = sw128_desc(smem_u32(s.a[st]), 16, 1024);
          const uint64_t db = sw128_desc(smem_u32(s.b[st]), 16, 1024);
          if (kb == kb0)
            umma_pair<false>(d, da, db, kIdesc);
          else
            umma_pair<true>(d, da, db, kIdesc);
          umma_pair<true>(d, da + 2, db + 2, kIdesc);
          umma_pair<true>(d, da + 4, db + 4, kIdesc);
          umma_pair<true>(d, da + 6, db + 6, kIdesc);
          umma_commit_pair(&s.empty[st]);
        }
        if (ok) umma_commit_pair(&s.acc_full[ab]);
      }
      asm volatile("tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                       smem_u32(&s.fin))
                   : "memory");
      mbar_wait(&s.fin, 0, p.err, nullptr);
    }
  } else {
    const int q = warp & 3;
    const int r = 32 * q + lane;
    uint32_t tc = 0;
    for (int t = pair; !s.abort && t < n_tiles; t += n_pairs, ++tc) {
      const uint32_t ab = tc & 1, use = tc >> 1;
      if (!warp_wait(&s.acc_full[ab], use & 1, p.err, abort_flag)) break;
      tc_fence_after();
      const int bt = t / p.split;
      const int m0 = (bt % tiles_m2) * 2 * BM + rank * BM, nb = bt / tiles_m2;
      const long long row = static_cast<long long>(m0) + r;
      const bool row_ok = row < M;
      const uint32_t acc = tmem + (static_cast<uint32_t>(32 * q) << 16) + ab * BN;
      if (p.split > 1) {
        // fp32 partial products of this slice (all 32 rows of the warp; rows
        // past M are never read): 32 x 32 blocks through the slabs, TMA
        // stores; the reduction kernel applies the epilogue
        const int prow = static_cast<int>((static_cast<long long>(t % p.split) * p.tiles_n + nb) * (tiles_m2 * 2 * BM) +
                                          m0 + 32 * q);
#pragma unroll 1
        for (int c = 0; c < BN; c += 64) {
          if (lane == 0) bulk_wait_read();
          __syncwarp();
          float v[32];
          load_acc32(acc + c, v);
          stage32_f32(s.epi[q][0], lane, v);
          load_acc32(acc + c + 32, v);
          stage32_f32(s.epi[q][1], lane, v);
          fence_proxy_async_smem();
          __syncwarp();
          if (lane == 0) {
            tma_store_2d(&tmap_part, s.epi[q][0], c, prow);
            tma_store_2d(&tmap_part, s.epi[q][1], c + 32, prow);
            bulk_commit();
          }
        }
      } else {
        const float rs = row_scale(p, row, row_ok);
        auto get = [&](int c, float (&v)[32]) {
          load_acc32(acc + c, v);
          if (p.rss) {
#pragma unroll
            for (int i = 0; i < 32; ++i) v[i] *= rs;
          }
        };
        const long long row0 = static_cast<long long>(m0) + 32 * q;
        if (row0 + 32 <= M)
          epilogue_warp_staged(p, &tmap_out, s.epi[q][0], s.epi[q][1], lane, row0, nb * BN, get);
        else
          epilogue_row(p, row, row_ok, nb * BN, get);
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) {
        if (rank == 0)
          mbar_arrive(&s.acc_empty[ab]);
        else
          remote_arrive(map_to_rank(&s.acc_empty[ab], 0));
      }
    }
    if (lane == 0) bulk_wait_all();
  }

  tc_fence_before();
  __syncthreads();
  cluster_sync_all();  // no CTA leaves while its peer may still signal it or read its operands
  if (warp == kWarpMma) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols2) : "memory");
  }
}

// Sum of the K slices' partials in slice order, then the epilogue: one warp
// per (row, 256-column block), lane l holding columns [8l, 8l + 8) (coalesced
// 1 KB per slice); the gated MLP pairs lane l with lane l + 16 (gate, up),
// the rotary embedding lane l with lane l ^ (D/16) (columns d, d + D/2).
__global__ void __launch_bounds__(256) split_reduce_kernel(Params p0) {
  pdl_launch_dependents();
  pdl_wait();
  const Params& p = p0;
  const long long M = rows_now(p);
  const int lane = threadIdx.x & 31;
  const long long w0 = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const long long nw = (static_cast<long long>(gridDim.x) * blockDim.x) >> 5;
  const long long mp = ((M + 2 * BM - 1) / (2 * BM)) * 2 * BM;
  for (long long u = w0; u < M * p.tiles_n; u += nw) {
    const int nb = static_cast<int>(u / M);
    const long long row = u % M;
    float v[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = 0.0f;
    for (int sl = 0; sl < p.split; ++sl) {
      const float4* src =
          reinterpret_cast<const float4*>(p.part + ((static_cast<long long>(sl) * p.tiles_n + nb) * mp + row) * BN) +
          2 * lane;
      const float4 a = __ldcg(src), b = __ldcg(src + 1);
      v[0] += a.x; v[1] += a.y; v[2] += a.z; v[3] += a.w;
      v[4] += b.x; v[5] += b.y; v[6] += b.z; v[7] += b.w;
    }
    if (p.rss) {
      const float rs = row_scale(p, row, true);
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] *= rs;
    }
    const int n0 = nb * BN;
    uint4 o;
    uint16_t* dst;
    bool write = true;
    if (p.epi == EPI_SWIGLU) {
      float up[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) up[i] = __shfl_down_sync(0xffffffffu, v[i], 16);
#pragma unroll
      for (int i = 0; i < 8; ++i) v[i] = silu(v[i]) * up[i];
      write = lane < 16;
      dst = p.out + row * p.ldo + n0 / 2 + 8 * lane;
    } else if (p.epi == EPI_ROPE && n0 < p.rope_cols) {
      const int half = p.head_dim / 2;
      float pv[8];
#pragma unroll
      for (int i = 0; i < 8; ++i) pv[i] = __shfl_xor_sync(0xffffffffu, v[i], half / 8);
      int lo = 0, hi = p.batch;  // largest b with cu[b] <= row
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (p.cu[mid] <= row) lo = mid; else hi = mid;
      }
      int pos = static_cast<int>(row - p.cu[lo]);
      if (pos >= p.max_pos) {
        if (lane == 0) raise_error(p.err, DEV_ERR_ARG);
        pos = p.max_pos - 1;
      }
      const bool first = (8 * lane) % p.head_dim < half;  // columns in the first half of the head
      const float2* tab = p.rope + static_cast<long long>((8 * lane) % half) * p.max_pos + pos;
#pragma unroll
      for (int i = 0; i < 8; ++i) {
        const float2 cs = tab[static_cast<long long>(i) * p.max_pos];
        v[i] = first ? v[i] * cs.x - pv[i] * cs.y : v[i] * cs.x + pv[i] * cs.y;
      }
      dst = p.out + row * p.ldo + n0 + 8 * lane;
    } else {
      dst = p.out + row * p.ldo + n0 + 8 * lane;
      if (p.epi == EPI_RESIDUAL) {
        const uint4 w = *reinterpret_cast<const uint4*>(p.residual + row * p.ldo + n0 + 8 * lane);
        v[0] += bf16lo(w.x); v[1] += bf16hi(w.x);
        v[2] += bf16lo(w.y); v[3] += bf16hi(w.y);
        v[4] += bf16lo(w.z); v[5] += bf16hi(w.z);
        v[6] += bf16lo(w.w); v[7] += bf16hi(w.w);
      }
    }
    o.x = pack_bf16x2(v[0], v[1]);
    o.y = pack_bf16x2(v[2], v[3]);
    o.z = pack_bf16x2(v[4], v[5]);
    o.w = pack_bf16x2(v[6], v[7]);
    if (write) *reinterpret_cast<uint4*>(dst) = o;
    if (p.ss_out && (p.epi == EPI_STORE || p.epi == EPI_RESIDUAL)) {
      float ss = sumsq8(o);  // lanes in order by a shuffle tree: a fixed order
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
      if (lane == 0) p.ss_out[row * p.tiles_n + nb] = ss;
    }
  }
}

// cos/sin table of the rotary embedding, frequency-major:
// tab[d][p] = (cos, sin)(p * theta^(-2d/D)).
__global__ void rope_table_kernel(float2* tab, int max_pos, int half, double theta) {
  pdl_launch_dependents();
  pdl_wait();
  const long long total = static_cast<long long>(max_pos) * half;
  for (long long q = static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x; q < total;
       q += static_cast<long long>(gridDim.x) * blockDim.x) {
    const int d = static_cast<int>(q / max_pos), pos = static_cast<int>(q % max_pos);
    const double ang = pos * pow(theta, -static_cast<double>(d) / half);
    tab[q] = make_float2(static_cast<float>(cos(ang)), static_cast<float>(sin(ang)));
  }
}

// Root-mean-square normalization of rows: one warp per row, fp32 sums.
// ANSWERS: only the last resp_len[b] rows of each request (rows below
// cu[b+1]), written packed in request order.
template <bool ANSWERS>
__global__ void __launch_bounds__(256) rmsnorm_kernel(const uint16_t* __restrict__ x, long long M, int C,
                                                      const uint16_t* __restrict__ gamma, float eps,
                                                      uint16_t* __restrict__ out, const int32_t* cu,
                                                      const int32_t* cu_resp, int batch,
                                                      const int32_t* __restrict__ rows_dev, unsigned* err) {
  pdl_launch_dependents();
  pdl_wait();
  if (rows_dev) M = clamp_rows(rows_dev, M, err);
  const int lane = threadIdx.x & 31;
  const long long w0 = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const long long nw = (static_cast<long long>(gridDim.x) * blockDim.x) >> 5;
  const int C8 = C / 8;
  for (long long o = w0; o < M; o += nw) {
    long long src = o;
    if constexpr (ANSWERS) {
      int lo = 0, hi = batch;  // request of answer row o: largest b with cu_resp[b] <= o
      while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (cu_resp[mid] <= o) lo = mid; else hi = mid;
      }
      const long long nresp = cu_resp[lo + 1] - cu_resp[lo];
      src = cu[lo + 1] - nresp + (o - cu_resp[lo]);
    }
    const uint4* xr = reinterpret_cast<const uint4*>(x + src * C);
    float ss = 0.f;
    for (int c = lane; c < C8; c += 32) {
      const uint4 v = xr[c];
      const float f[8] = {bf16lo(v.x), bf16hi(v.x), bf16lo(v.y), bf16hi(v.y),
                          bf16lo(v.z), bf16hi(v.z), bf16lo(v.w), bf16hi(v.w)};
#pragma unroll
      for (int i = 0; i < 8; ++i) ss = fmaf(f[i], f[i], ss);
    }
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xffffffffu, ss, off);
    const float inv = rsqrtf(ss / static_cast<float>(C) + eps);
    const uint4* gr = reinterpret_cast<const uint4*>(gamma);
    uint4* orow = reinterpret_cast<uint4*>(out + o * C);
    for (int c = lane; c < C8; c += 32) {
      const uint4 v = xr[c], g = gr[c];
      uint4 w;
      w.x = pack_bf16x2(bf16lo(v.x) * inv * bf16lo(g.x), bf16hi(v.x) * inv * bf16hi(g.x));
      w.y = pack_bf16x2(bf16lo(v.y) * inv * bf16lo(g.y), bf16hi(v.y) * inv * bf16hi(g.y));
      w.z = pack_bf16x2(bf16lo(v.z) * inv * bf16lo(g.z), bf16hi(v.z) * inv * bf16hi(g.z));
      w.w = pack_bf16x2(bf16lo(v.w) * inv * bf16lo(g.w), bf16hi(v.w) * inv * bf16hi(g.w));
      orow[c] = w;
    }
  }
}

// Sum of squares of each row's bf16 values (fp32, one warp per row, lanes in
// a shuffle tree): the normalization input of the first projection.
__global__ void __launch_bounds__(256) row_sumsq_kernel(const uint16_t* __restrict__ x, long long M, int C,
                                                        float* __restrict__ ss, const int32_t* __restrict__ rows_dev,
                                                        unsigned* err) {
  pdl_launch_dependents();
  pdl_wait();
  if (rows_dev) M = clamp_rows(rows_dev, M, err);
  const int lane = threadIdx.x & 31;
  const long long w0 = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const long long nw = (static_cast<long long>(gridDim.x) * blockDim.x) >> 5;
  const int C8 = C / 8;
  for (long long r = w0; r < M; r += nw) {
    const uint4* xr = reinterpret_cast<const uint4*>(x + r * C);
    float s = 0.0f;
    for (int c = lane; c < C8; c += 32) s += sumsq8(xr[c]);
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) s += __shfl_xor_sync(0xffffffffu, s, off);
    if (lane == 0) ss[r] = s;
  }
}

// Answer rows of the step input from the embedding table: row
// cu[b+1] - resp[b] + i of request b is table[tokens[cu_resp[b] + i]], or
// table[mask_id] while that position is still masked (token < 0).
__global__ void __launch_bounds__(256) embed_answers_kernel(const uint16_t* __restrict__ table, int V, int C,
                                                            const int32_t* __restrict__ tokens, int mask_id,
                                                            const int32_t* cu, const int32_t* cu_resp, int batch,
                                                            long long R, uint16_t* __restrict__ x,
                                                            unsigned* err) {
  pdl_launch_dependents();
  pdl_wait();
  const int lane = threadIdx.x & 31;
  const long long w0 = (static_cast<long long>(blockIdx.x) * blockDim.x + threadIdx.x) >> 5;
  const long long nw = (static_cast<long long>(gridDim.x) * blockDim.x) >> 5;
  const int C8 = C / 8;
  for (long long o = w0; o < R; o += nw) {
    int lo = 0, hi = batch;
    while (hi - lo > 1) {
      const int mid = (lo + hi) >> 1;
      if (cu_resp[mid] <= o) lo = mid; else hi = mid;
    }
    const long long nresp = cu_resp[lo + 1] - cu_resp[lo];
    const long long dst = cu[lo + 1] - nresp + (o - cu_resp[lo]);
    int tok = tokens[o];
    if (tok < 0) tok = mask_id;
    if (tok >= V) {
      if (lane == 0) raise_error(err, DEV_ERR_ARG);
      tok = mask_id;
    }
    const uint4* src = reinterpret_cast<const uint4*>(table + static_cast<long long>(tok) * C);
    uint4* d = reinterpret_cast<uint4*>(x + dst * C);
    for (int c = lane; c < C8; c += 32) d[c] = src[c];
  }
}

}  // namespace gemm
}  // namespace davet

using namespace davet;
using namespace davet::gemm;

namespace {

using EncodeTiledFn = CUresult (*)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*, const cuuint64_t*,
                                   const cuuint64_t*, const cuuint32_t*, const cuuint32_t*, CUtensorMapInterleave,
                                   CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
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

// 2-D map over a row-major bf16 [rows][K] matrix, boxes of 64 x box_rows.
bool make_map(CUtensorMap* m, const void* base, long long rows, int K, int box_rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(K), static_cast<cuuint64_t>(std::max<long long>(rows, 1))};
  const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(K) * 2};
  const cuuint32_t box[2] = {static_cast<cuuint32_t>(BK), static_cast<cuuint32_t>(box_rows)};
  const cuuint32_t estride[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), gdim, gstride, box, estride,
             CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

int g_sms[64] = {0};
bool g_attr[64] = {false};
std::mutex g_mu;

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }


// K slices for the CTA-pair kernel when its tiles cover less than half of the
// pairs (few rows and few column blocks): as many slices as fill the pairs,
// each at least 8 k-blocks.  1 = no split.
int pick_split(long long M, int tiles_n, int nk, int pairs) {
  if (M <= BM) return 1;
  const long long tiles2 = ((M + 2 * BM - 1) / (2 * BM)) * tiles_n;
  if (2 * tiles2 > pairs) return 1;
  const int S = std::min(static_cast<int>(pairs / tiles2), nk / 8);
  return S >= 2 ? S : 1;
}

// fp32 partial rows: [S][tiles_n][M rounded up to 256][256]
long long split_rows(long long M, int tiles_n, int S) {
  return static_cast<long long>(S) * tiles_n * (((M + 2 * BM - 1) / (2 * BM)) * 2 * BM);
}
size_t split_bytes(long long M, int tiles_n, int S) { return static_cast<size_t>(split_rows(M, tiles_n, S)) * BN * 4; }

// 2-D map over the fp32 partial rows [rows][256], boxes of 32 x 32.
bool make_part_map(CUtensorMap* m, void* base, long long rows) {
  EncodeTiledFn enc = encode_fn();
  if (!enc) return false;
  const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(BN), static_cast<cuuint64_t>(rows)};
  const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(BN) * 4};
  const cuuint32_t box[2] = {32, 32};
  const cuuint32_t estride[2] = {1, 1};
  return enc(m, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, base, gdim, gstride, box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
             CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
             CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace

extern "C" davet_status davet_linear_workspace_bytes(int64_t M, int K, int N, size_t* bytes) {
  if (!bytes || M < 0 || K < BK || K % BK != 0 || N < BN || N % BN != 0) return DAVET_ERR_INVALID_ARG;
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  if (dev < 0 || dev >= 64) return DAVET_ERR_UNSUPPORTED;
  int sms = 0;
  e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return cuda_fail(e);
  const int S = pick_split(M, N / BN, K / BK, sms / 2);
  *bytes = S > 1 ? split_bytes(M, N / BN, S) : 0;
  return DAVET_OK;
}

extern "C" davet_status davet_linear(const void* A, int64_t M, int K, const void* W, int N, void* out, int epilogue,
                                     const void* residual, const int32_t* cu_seqlens, int batch, int rope_cols,
                                     int head_dim, const void* rope_table, int max_pos, void* workspace,
                                     size_t workspace_bytes, const float* row_ss, int row_ss_parts, float row_ss_eps,
                                     float* ss_out, const int32_t* rows_dev, void* stream) {
  if (M < 0 || M > 0x7fffffffLL || K < BK || K % BK != 0 || N < BN || N % BN != 0) return DAVET_ERR_INVALID_ARG;
  if (epilogue < EPI_STORE || epilogue > EPI_ROPE) return DAVET_ERR_INVALID_ARG;
  if (row_ss && (row_ss_parts < 1 || !(row_ss_eps >= 0.0f))) return DAVET_ERR_INVALID_ARG;
  if (ss_out && epilogue != EPI_STORE && epilogue != EPI_RESIDUAL) return DAVET_ERR_INVALID_ARG;
  if (M == 0) return DAVET_OK;
  if (!A || !W || !out || !aligned16(A) || !aligned16(W) || !aligned16(out)) return DAVET_ERR_INVALID_ARG;
  if (epilogue == EPI_RESIDUAL && (!residual || !aligned16(residual))) return DAVET_ERR_INVALID_ARG;
  if (epilogue == EPI_ROPE) {
    if (!cu_seqlens || batch < 1 || !rope_table || max_pos < 1 || (head_dim != 64 && head_dim != 128) ||
        rope_cols < 0 || rope_cols % BN != 0 || rope_cols > N)
      return DAVET_ERR_INVALID_ARG;
  }
  int dev = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_fail(e);
  if (dev < 0 || dev >= 64) return DAVET_ERR_UNSUPPORTED;
  const size_t smem = sizeof(Smem) + 1024;
  const size_t smem2 = sizeof(Smem2) + 1024;
  {
    std::lock_guard<std::mutex> g(g_mu);
    if (g_sms[dev] == 0) {
      e = cudaDeviceGetAttribute(&g_sms[dev], cudaDevAttrMultiProcessorCount, dev);
      if (e != cudaSuccess) return cuda_fail(e);
    }
    if (!g_attr[dev]) {
      e = cudaFuncSetAttribute(gemm_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
      if (e == cudaSuccess)
        e = cudaFuncSetAttribute(gemm2_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem2));
      if (e != cudaSuccess) return cuda_fail(e);
      g_attr[dev] = true;
    }
  }
  unsigned* err = device_error_word();
  if (!err) return DAVET_ERR_CUDA;
  CUtensorMap ma, mw;
  // the output map: boxes of 32 rows x 64 columns (one epilogue warp's slab)
  CUtensorMap mo;
  if (!make_map(&ma, A, M, K, BM) || !make_map(&mw, W, N, K, BN) ||
      !make_map(&mo, out, M, epilogue == EPI_SWIGLU ? N / 2 : N, 32))
    return DAVET_ERR_INVALID_ARG;
  Params p;
  p.M = M;
  p.N = N;
  p.K = K;
  p.tiles_m = static_cast<int>((M + BM - 1) / BM);
  p.tiles_n = N / BN;
  p.out = static_cast<uint16_t*>(out);
  p.ldo = epilogue == EPI_SWIGLU ? N / 2 : N;
  p.residual = static_cast<const uint16_t*>(residual);
  p.epi = epilogue;
  p.cu = cu_seqlens;
  p.batch = batch;
  p.rope_cols = epilogue == EPI_ROPE ? rope_cols : 0;
  p.head_dim = head_dim;
  p.max_pos = max_pos;
  p.rope = static_cast<const float2*>(rope_table);
  p.err = err;
  p.split = 1;
  p.kb_per = K / BK;
  p.part = nullptr;
  p.rows_dev = rows_dev;
  p.rss = row_ss;
  p.rss_parts = row_ss ? row_ss_parts : 0;
  p.rss_eps = row_ss_eps;
  p.ss_out = ss_out;
  const long long tiles = static_cast<long long>(p.tiles_m) * p.tiles_n;
  if (tiles > 0x7fffffffLL) return DAVET_ERR_UNSUPPORTED;
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  // 256 x 256 tiles on CTA pairs whenever the odd CTA has rows to compute:
  // the same work per SM as 128 x 256 tiles, half the operand bytes per SM
  const int pairs = g_sms[dev] / 2;
  const long long tiles2 = ((M + 2 * BM - 1) / (2 * BM)) * p.tiles_n;
  if (M > BM) {
    CUtensorMap mw2, mp;
    if (!make_map(&mw2, W, N, K, BM)) return DAVET_ERR_INVALID_ARG;
    mp = mo;  // the partial map is read only with a split
    const int S = pick_split(M, p.tiles_n, K / BK, pairs);
    if (S > 1 && workspace && workspace_bytes >= split_bytes(M, p.tiles_n, S) && aligned16(workspace)) {
      if (!make_part_map(&mp, workspace, split_rows(M, p.tiles_n, S))) return DAVET_ERR_INVALID_ARG;
      p.split = S;
      p.kb_per = (K / BK) / S;
      p.part = static_cast<float*>(workspace);
    }
    const int grid2 = 2 * static_cast<int>(std::min<long long>(tiles2 * p.split, pairs));
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(grid2);
    cfg.blockDim = dim3(kThreads);
    cfg.dynamicSmemBytes = smem2;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = pdl_enabled() ? 2 : 1;
    e = cudaLaunchKernelEx(&cfg, gemm2_kernel, ma, mw2, mo, mp, p);
    if (e != cudaSuccess) return cuda_fail(e);
    if (p.split > 1) {
      const long long warps = M * p.tiles_n;
      const unsigned blocks = static_cast<unsigned>(std::min<long long>((warps + 7) / 8, 152LL * 16));
      e = launch(split_reduce_kernel, dim3(blocks), dim3(256), 0, st, p);
      if (e != cudaSuccess) return cuda_fail(e);
    }
    return check_launch();
  }
  const int grid = static_cast<int>(std::min<long long>(tiles, g_sms[dev]));
  e = launch(gemm_kernel, dim3(grid), dim3(kThreads), smem, st, ma, mw, mo, p);
  if (e != cudaSuccess) return cuda_fail(e);
  return check_launch();
}

extern "C" davet_status davet_rope_table(int max_pos, int head_dim, double theta, void* table, void* stream) {
  if (max_pos < 1 || (head_dim != 64 && head_dim != 128) || !(theta > 1.0) || !table) return DAVET_ERR_INVALID_ARG;
  const long long total = static_cast<long long>(max_pos) * (head_dim / 2);
  const int blocks = static_cast<int>(std::min<long long>((total + 255) / 256, 152LL * 8));
  const cudaError_t e = launch(rope_table_kernel, dim3(blocks), dim3(256), 0, static_cast<cudaStream_t>(stream),
                               static_cast<float2*>(table), max_pos, head_dim / 2, theta);
  if (e != cudaSuccess) return cuda_fail(e);
  return check_launch();
}

extern "C" davet_status davet_rmsnorm(const void* x, int64_t M, int C, const void* gamma, float eps, void* out,
                                      const int32_t* cu_seqlens, const int32_t* cu_resp, int batch,
                                      const int32_t* rows_dev, void* stream) {
  if (M < 0 || C < 8 || C % 8 != 0 || !(eps >= 0.0f)) return DAVET_ERR_INVALID_ARG;
  if (M == 0) return DAVET_OK;
  if (!x || !gamma || !out || !aligned16(x) || !aligned16(gamma) || !aligned16(out)) return DAVET_ERR_INVALID_ARG;
  const bool answers = cu_resp != nullptr;
  if (answers && (!cu_seqlens || batch < 1)) return DAVET_ERR_INVALID_ARG;
  unsigned* err = device_error_word();
  if (!err) return DAVET_ERR_CUDA;
  const int blocks = static_cast<int>(std::min<long long>((M + 7) / 8, 152LL * 16));
  cudaStream_t st = static_cast<cudaStream_t>(stream);
  const uint16_t* xs = static_cast<const uint16_t*>(x);
  const uint16_t* gs = static_cast<const uint16_t*>(gamma);
  uint16_t* os = static_cast<uint16_t*>(out);
  const cudaError_t e =
      answers ? launch(rmsnorm_kernel<true>, dim3(blocks), dim3(256), 0, st, xs, static_cast<long long>(M), C, gs, eps,
                       os, cu_seqlens, cu_resp, batch, rows_dev, err)
              : launch(rmsnorm_kernel<false>, dim3(blocks), dim3(256), 0, st, xs, static_cast<long long>(M), C, gs,
                       eps, os, cu_seqlens, cu_resp, batch, rows_dev, err);
  if (e != cudaSuccess) return cuda_fail(e);
  return check_launch();
}

extern "C" davet_status davet_row_sumsq(const void* x, int64_t M, int C, float* ss_out, const int32_t* rows_dev,
                                         void* stream) {
  if (M < 0 || C < 8 || C % 8 != 0) return DAVET_ERR_INVALID_ARG;
  if (M == 0) return DAVET_OK;
  if (!x || !ss_out || !aligned16(x)) return DAVET_ERR_INVALID_ARG;
  unsigned* err = device_error_word();
  if (!err) return DAVET_ERR_CUDA;
  const int blocks = static_cast<int>(std::min<long long>((M + 7) / 8, 152LL * 16));
  const cudaError_t e = launch(row_sumsq_kernel, dim3(blocks), dim3(256), 0, static_cast<cudaStream_t>(stream),
                               static_cast<const uint16_t*>(x), static_cast<long long>(M), C, ss_out, rows_dev, err);
  if (e != cudaSuccess) return cuda_fail(e);
  return check_launch();
}

extern "C" davet_status davet_embed_answers(const void* table, int V, int C, const int32_t* tokens, int mask_id,
                                            const int32_t* cu_seqlens, const int32_t* cu_resp, int batch,
                                            int64_t total_resp, void* x, void* stream) {
  if (V < 1 || C < 8 || C % 8 != 0 || mask_id < 0 || mask_id >= V || batch < 1 || total_resp < 0)
    return DAVET_ERR_INVALID_ARG;
  if (total_resp == 0) return DAVET_OK;
  if (!table || !tokens || !cu_seqlens || !cu_resp || !x || !aligned16(table) || !aligned16(x))
    return DAVET_ERR_INVALID_ARG;
  unsigned* err = device_error_word();
  if (!err) return DAVET_ERR_CUDA;
  const int blocks = static_cast<int>(std::min<long long>((total_resp + 7) / 8, 152LL * 16));
  const cudaError_t e = launch(embed_answers_kernel, dim3(blocks), dim3(256), 0, static_cast<cudaStream_t>(stream),
                               static_cast<const uint16_t*>(table), V, C, tokens, mask_id, cu_seqlens, cu_resp, batch,
                               static_cast<long long>(total_resp), static_cast<uint16_t*>(x), err);
  if (e != cudaSuccess) return cuda_fail(e);
  return check_launch();
}
