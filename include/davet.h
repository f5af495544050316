/*
 * davet.h -- C ABI of the GB300 (sm_103a) DAVET step-conditioning library.
 *
 * DAVET (Denoising-Aware Visual Evidence Trajectory allocation) conditions
 * every denoising step of a diffusion vision-language model on one view of
 * an ordered hierarchy of visual "evidence views" built once from a single
 * visual encoding (Sec. 4.3).  This library implements the data-parallel
 * path that the policy drives:
 *
 *   davet_build_pyramid   the evidence hierarchy (Sec. 4.3), once per request
 *   davet_gather_view     the step input [view || prompt || answer] (Eq. 5),
 *                         the view a pooled level or the mixed view
 *   davet_step_attention  bidirectional attention over it (Sec. 3.1, Eq. 1)
 *   davet_build_views     every view once as a contiguous [view || text] block
 *   davet_build_views_pruned, davet_build_views_merged   the same blocks from
 *                         the pruning and merging realizers (Sec. 4.3, 5.3)
 *   davet_view_attention  the gather and the attention fused: attention reads
 *                         each request's step sequence from its view block
 *   davet_unmask_topk     argmax, confidence and confidence-ranked commit
 *                         (Sec. 3.1, Eq. 1-2) plus the mean confidence and
 *                         churn that drive the trajectory risk (Eq. 7)
 *   davet_policy_*        the allocation policy that picks each step's view
 *                         (Sec. 4.2, Eq. 6-8; Sec. 4.3, Eq. 9)
 *   davet_linear, davet_rmsnorm, davet_rope_table, davet_embed_answers
 *                         the dense part of a full backbone layer step
 *                         (tcgen05 GEMM with fused epilogues)
 *
 * Conventions shared by every entry point:
 *  - Pointers named *_dev, and every tensor argument, are DEVICE pointers on
 *    the device current to the calling thread (davet_unmask_topk's logits may
 *    also be device-addressable pinned host memory).  The caller owns every buffer;
 *    the library never allocates, frees or retains caller memory.
 *  - bf16 tensors are IEEE bfloat16 bit patterns (uint16), row-major, with
 *    the layout given per function.  Tensor base pointers must be 16-byte
 *    aligned.
 *  - `stream` is a cudaStream_t (NULL = the legacy default stream).  Every
 *    call only enqueues work on that stream and returns without waiting.
 *    davet_build_pyramid, davet_gather_view, davet_step_attention,
 *    davet_view_attention and davet_unmask_topk never synchronize the host, so they can be captured in
 *    a CUDA graph once each has run at least once on the device outside of a
 *    capture (the first call per device resolves a few device addresses).
 *  - Host-visible argument checks run before anything is enqueued and return
 *    DAVET_ERR_INVALID_ARG or DAVET_ERR_UNSUPPORTED.  A failed launch returns
 *    DAVET_ERR_CUDA (the CUDA error code is kept for davet_last_cuda_error).
 *  - Values that live on the device (lengths, levels) are checked by the
 *    kernels: an out-of-range value never leads to an out-of-bounds access;
 *    instead the kernel clamps, skips the offending item and sets a bit in a
 *    per-device error word that davet_device_status() reads.  Device-side
 *    waits are bounded; a wait that gives up sets the timeout bit and the
 *    kernel returns early (its outputs are then undefined).
 *  - No C++ exception crosses this interface.
 */
#ifndef DAVET_H_
#define DAVET_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum davet_status {
  DAVET_OK = 0,
  DAVET_ERR_INVALID_ARG = 1, /* null pointer, bad size, misalignment */
  DAVET_ERR_UNSUPPORTED = 2, /* valid request outside the supported shapes */
  DAVET_ERR_CUDA = 3,        /* a CUDA runtime call or launch failed */
  DAVET_ERR_TIMEOUT = 4,     /* device error word: a bounded wait gave up */
  DAVET_ERR_DEVICE = 5       /* device error word: capacity or argument bit set */
} davet_status;

/* Device error word bits (davet_device_status). */
#define DAVET_DEV_TIMEOUT 0x1u  /* a kernel's bounded wait gave up */
#define DAVET_DEV_CAPACITY 0x2u /* a device-side length exceeded a capacity */
#define DAVET_DEV_ARG 0x4u      /* a device-side argument was out of range */

/* Library version, major * 10000 + minor * 100 + patch. */
int davet_version(void);

/* Static, NUL-terminated description of a status code (never NULL). */
const char* davet_status_string(int status);

/* The cudaError_t recorded by the last call on this thread that returned
 * DAVET_ERR_CUDA (0 if none). */
int davet_last_cuda_error(void);

/*
 * Reads the device error word of the current device into *flags (bits
 * DAVET_DEV_*), optionally clearing it.  This call SYNCHRONIZES the device
 * (it copies the word to the host); call it outside stream capture.
 * Returns DAVET_OK when no bit is set, DAVET_ERR_TIMEOUT when the timeout
 * bit is set, DAVET_ERR_DEVICE when another bit is set.
 */
davet_status davet_device_status(unsigned* flags, int clear);

/*
 * The same word read on `stream`: waits for the work queued on that stream
 * only (not the whole device), copies the word to *flags (nullable) and
 * returns DAVET_OK, DAVET_ERR_TIMEOUT or DAVET_ERR_DEVICE as above.  It does
 * not clear the word.  Outside stream capture.
 */
davet_status davet_sync_status(void* stream, unsigned* flags);

/*
 * Diagnostic of the failure path: one thread waits, with the bounded wait
 * every kernel of the library uses, on an mbarrier that nothing signals.
 * After the wait budget (about a second of SM clocks) it gives up, raises
 * DAVET_DEV_TIMEOUT in the device error word and writes 1 to *gave_up_dev
 * (int32, device); the context stays usable.  Nothing else uses it.
 */
davet_status davet_selftest_wait_timeout(int* gave_up_dev, void* stream);

/* --------------------------------------------------------- evidence views */

/*
 * Host-only layout helper for the evidence pyramid (Sec. 4.3: an ordered
 * hierarchy of views built from one encoding by structured pooling; the
 * finest view is the encoding itself).
 *   grid       side G of each square tile of visual tokens (>= 1)
 *   n_levels   number of levels, 1..5; level 0 is the unpooled grid and
 *              G_l = ceil(G_{l-1} / 2)
 *   n_tiles    tiles of the request (>= 0)
 *   level_side[n_levels]         out (nullable): G_l
 *   level_row_offset[n_levels+1] out (nullable): first row of each level in
 *              the level-major pyramid layout; [n_levels] is the total row
 *              count.  Within a level, rows are tile-major, then row-major
 *              within a tile: row = offset[l] + t*G_l^2 + y*G_l + x.
 */
davet_status davet_pyramid_layout(int grid, int n_levels, int n_tiles, int* level_side,
                                  int64_t* level_row_offset);

/*
 * Builds the evidence pyramid of one request (Sec. 4.3, "structured
 * pooling", all views constructed once before denoising).  Level l >= 1
 * cell (y, x) is the mean of the level l-1 cells (2y+i, 2x+j), i, j in
 * {0, 1}, that lie inside the level l-1 grid (a 2x2 stride-2 cascade; edge
 * cells of odd grids average their in-range children only).  Accumulation
 * is fp32 from the level below held in fp32; each level is rounded to bf16
 * once, on store.
 *   feat     bf16 [n_tiles][grid][grid][C], the encoding (level 0)
 *   pyr      bf16 [level_row_offset[n_levels]][C], level-major layout of
 *            davet_pyramid_layout.  If pyr == feat, level 0 is already in
 *            place and only levels >= 1 are written; otherwise feat must not
 *            overlap pyr and level 0 is copied into pyr as well.
 *   C        channels per token, a multiple of 8
 *   pyr_f32  nullable fp32 [level_row_offset[n_levels]][C]: every level
 *            before rounding (level 0 widened exactly)
 * n_tiles == 0 is a no-op.
 */
davet_status davet_build_pyramid(const void* feat, void* pyr, int n_tiles, int grid, int n_levels, int C,
                                 float* pyr_f32, void* stream);

/*
 * Host-only layout helper for the mixed evidence view (Sec. 4.3: the pooled
 * representation augmented with a fixed subset of unpooled tokens).  The
 * paper does not fix the subset; this library takes, per tile, every row of
 * pyramid level mixed_level followed by the level-0 tokens of a centred
 * stride-s lattice, (y, x) with y, x in {s/2, s/2 + s, s/2 + 2s, ...} below
 * grid, in row-major order.
 *   grid, n_levels   as for davet_pyramid_layout
 *   mixed_level      the pooled level, 0 <= mixed_level < n_levels
 *   mixed_stride     s, 1 <= s <= grid
 *   rows_per_tile    out (nullable): G_{mixed_level}^2 + n^2 with
 *                    n = ceil((grid - s/2) / s)
 * Example: grid 27, 4 levels, level 2 and s = 3 give 49 + 81 = 130 rows.
 */
davet_status davet_mixed_view_rows(int grid, int n_levels, int mixed_level, int mixed_stride,
                                   int* rows_per_tile);

/*
 * Packs the input of one denoising step for a batch of requests (Eq. 5:
 * the step is conditioned on v_t = A(v; b_t), the view selected for the
 * step, together with the query and the current answer state).  For request
 * b the packed rows are
 *     [ all rows of view level_dev[b] of its pyramid (tiles in order)
 *       || its prompt_len_dev[b] prompt rows || its resp_len_dev[b] answer rows ]
 * and requests follow one another in batch order.  View l < n_levels is
 * pyramid level l; view n_levels is the mixed view of
 * davet_mixed_view_rows (tile by tile, its rows are read straight from the
 * pyramid, nothing is stored for it).  Rows are copied bit for bit.
 * cu_seqlens_dev[b] receives the first packed row of request b and
 * cu_seqlens_dev[batch] the total row count.
 *   pyr_ptrs_dev     device array [batch] of device pointers to each
 *                    request's bf16 pyramid (davet_build_pyramid layout)
 *   tiles_dev        int32 [batch] tiles per request
 *   text             bf16 [*][C]; request b's prompt and answer rows are
 *                    contiguous from row text_off_dev[b] (int64 [batch])
 *   prompt_len_dev, resp_len_dev, level_dev   int32 [batch]
 *   grid, n_levels, C  as for davet_build_pyramid (shared by the batch)
 *   mixed_level, mixed_stride  the mixed view (as for davet_mixed_view_rows);
 *                    mixed_stride = 0 means the batch has no mixed view
 *   packed           bf16 [max_total_rows][C] output
 *   cu_seqlens_dev   int32 [batch+1] output
 * Device-side checks: a level outside [0, n_levels) (or [0, n_levels] with
 * a mixed view) or a negative count sets DAVET_DEV_ARG and the request
 * contributes no visual rows; a total above
 * max_total_rows sets DAVET_DEV_CAPACITY, rows beyond the capacity are not
 * written and cu_seqlens is clamped to max_total_rows.
 */
davet_status davet_gather_view(const void* const* pyr_ptrs_dev, const int32_t* tiles_dev, const void* text,
                               const int64_t* text_off_dev, const int32_t* prompt_len_dev,
                               const int32_t* resp_len_dev, const int32_t* level_dev, int batch, int grid,
                               int n_levels, int mixed_level, int mixed_stride, int C, void* packed,
                               int32_t* cu_seqlens_dev, int64_t max_total_rows, void* stream);

/* ------------------------------------------------------- step attention */

/*
 * Bidirectional multi-head attention of one denoising step (Sec. 3.1, Eq. 1:
 * masked positions are predicted in parallel through bidirectional
 * attention).  For every request b, every row i of the request and head h:
 *     out[i][h] = sum_j softmax_j(scale * q_i,h . k_j,h) v_j,h
 * over all rows j of the same request (no causal mask, no attention across
 * requests).  tcgen05 tensor-core kernel; bf16 inputs, fp32 accumulation and
 * softmax, bf16 output.
 *   qkv             bf16 [max_total_rows][3][H][D]: per row the query, key
 *                   and value of every head (the packed rows of
 *                   davet_gather_view with C = 3*H*D)
 *   cu_seqlens_dev  int32 [batch+1] request boundaries, non-decreasing,
 *                   cu[0] = 0, cu[batch] <= max_total_rows
 *   H >= 1, D in {64, 128}, scale > 0 (usually 1/sqrt(D))
 *   out             bf16 [max_total_rows][H][D]; rows past cu[batch] are not
 *                   written
 * Device-side checks: boundaries outside [0, max_total_rows] or decreasing
 * set DAVET_DEV_ARG and are clamped.
 */
davet_status davet_step_attention(const void* qkv, const int32_t* cu_seqlens_dev, int batch,
                                  int64_t max_total_rows, int H, int D, float scale, void* out, void* stream);

/*
 * Scratch of davet_step_attention and davet_view_attention: *bytes = 0 (each
 * CTA builds the request schedule in its shared memory), for callers that
 * size a workspace per call.  DAVET_ERR_INVALID_ARG for a negative size or a
 * null `bytes`, DAVET_ERR_UNSUPPORTED for D other than 64 or 128.
 */
davet_status davet_step_attention_workspace(int batch, int64_t max_total_rows, int H, int D, size_t* bytes);

/*
 * View blocks (host-only helpers and the build).  In the view-block layout a
 * request keeps every evidence view once as a contiguous block
 *     [ view rows (n_tiles * rows_per_tile[v]) || its text_rows prompt and
 *       answer rows ]
 * for views v = 0..n_views-1: the pooled levels 0..n_levels-1 (Sec. 4.3,
 * rows as in davet_pyramid_layout) and, when mixed_stride != 0, the mixed
 * view as view n_levels (davet_mixed_view_rows).  A step's input for view v
 * (Eq. 5) is then one run of rows, which davet_view_attention reads directly.
 *
 * davet_view_rows: rows_per_tile (int [n_views], nullable) and n_views (int*,
 * nullable) for this geometry.
 * davet_view_layout: block_row0 (int64 [n_views + 1], nullable): first row of
 * each block within the request's buffer; [n_views] is the buffer's rows.
 */
davet_status davet_view_rows(int grid, int n_levels, int mixed_level, int mixed_stride, int* rows_per_tile,
                             int* n_views);
davet_status davet_view_layout(int grid, int n_levels, int mixed_level, int mixed_stride, int n_tiles, int text_rows,
                               int64_t* block_row0);

/*
 * Builds one request's view blocks (Sec. 4.3: all views constructed once
 * before denoising): the pooled levels as davet_build_pyramid defines them
 * (level l at the start of block l), the mixed view's rows, and a copy of the
 * request's text rows in every block.
 *   feat   bf16 [n_tiles][grid][grid][C]; if feat == buf the encoding is
 *          already in place at the start of block 0, otherwise it is copied
 *          there (feat must not overlap buf then)
 *   buf    bf16 [block_row0[n_views]][C], the request's buffer
 *   text   bf16 [text_rows][C], the prompt and answer rows; must not overlap
 *          buf (nullable when text_rows == 0)
 * Enqueues two kernels on `stream`.
 */
davet_status davet_build_views(const void* feat, void* buf, const void* text, int n_tiles, int grid, int n_levels,
                               int mixed_level, int mixed_stride, int text_rows, int C, void* stream);

/*
 * Alternative evidence realizers (Sec. 4.3 "compatible evidence realizers":
 * pruning varies the retention ratio, merging the aggregation strength;
 * Sec. 5.3 / Table 2 runs the same allocation policy over pooling, pruning and
 * merging).  Each builds the same view blocks as davet_build_views -- the
 * same views, rows per tile (davet_view_rows), layout (davet_view_layout)
 * and text rows -- so davet_view_attention reads them unchanged; only the
 * rows of the views differ.  feat, buf, text and the geometry arguments are
 * as for davet_build_views; grid <= 64 and n_tiles <= 65535 (else
 * DAVET_ERR_UNSUPPORTED).
 *
 * davet_build_views_pruned -- nested visual-token pruning.  The paper leaves
 * the importance score open; it is an input:
 *   score  fp32 [n_tiles][grid*grid], device, the score of each token (raster
 *          order) of each tile; a NaN ranks below every number
 * View v keeps, per tile, the davet_view_rows(v) highest-scoring tokens
 * (equal scores by ascending index) in raster order, so every view is a
 * subset of each larger one; the mixed view, if any, is the one of that
 * length.  DAVET_ERR_INVALID_ARG if a view has more rows per tile than a tile
 * has tokens.  Enqueues two kernels.
 *
 * davet_build_views_merged -- hierarchical similarity merging.  Level 0 is
 * the encoding; level l is built from level l-1 by bipartite matching rounds
 * (positions 0, 2, 4, ... form set A, 1, 3, 5, ... set B; each member of A is
 * matched to the member of B of highest cosine similarity, ties to the
 * smaller B; the r = min(n - G_l^2, ceil(n/2)) best-matched members of A,
 * ties to the smaller position, merge into their match; survivors keep their
 * order) until it holds G_l^2 tokens, the pooled level's count.  Similarity
 * is measured on channels [sim_c0, sim_c0 + sim_C) of the token's feature
 * sum; each merged row is the mean of the level-0 rows it absorbed.  All of
 * it is binary32 in a fixed order: feature sums add the members in ascending
 * level-0 index, dot products and squared norms are fused multiply-add
 * chains in ascending channel order, 1/|s| is a correctly rounded square
 * root then division (0 for a zero vector), sim = (dot * 1/|a|) * 1/|b|, a
 * row is sum / count correctly rounded then rounded to bf16 (nearest even).
 * The mixed view, if any, is the merged coarse level plus the level-0
 * lattice, as for pooling.  Inputs must be finite.
 *   sim_c0, sim_C   similarity channels: sim_c0 % 8 == 0, sim_C % 32 == 0,
 *                   sim_c0 + sim_C <= C
 *   assign          int32 [n_levels][n_tiles][grid*grid], device, nullable:
 *                   the level-l token each level-0 token belongs to
 *   workspace       device, 256-byte aligned, davet_merge_workspace_bytes
 *                   bytes; not read before it is written
 * Enqueues three launches per round and one per level on `stream`.
 */
davet_status davet_build_views_pruned(const void* feat, const float* score, void* buf, const void* text, int n_tiles,
                                      int grid, int n_levels, int mixed_level, int mixed_stride, int text_rows, int C,
                                      void* stream);
davet_status davet_merge_workspace_bytes(int n_tiles, int grid, int n_levels, int sim_C, size_t* bytes);
davet_status davet_build_views_merged(const void* feat, void* buf, const void* text, int n_tiles, int grid,
                                      int n_levels, int mixed_level, int mixed_stride, int text_rows, int C,
                                      int sim_c0, int sim_C, int32_t* assign, void* workspace,
                                      size_t workspace_bytes, void* stream);

/*
 * davet_gather_view followed by davet_step_attention in one kernel (Eq. 5,
 * then Sec. 3.1, Eq. 1), without the packed step input: request b's sequence
 * [view || prompt || answer] for its step view is the view block that
 * davet_build_views laid out, and the attention kernel reads its query, key
 * and value rows straight from it.  out and cu_seqlens_dev are what
 * davet_gather_view + davet_step_attention produce for the same views.
 *   store            bf16 [store_rows][3][H][D]: every request's view-block
 *                    buffer (C = 3*H*D)
 *   buf_row0_dev     int64 [batch]: first store row of request b's buffer
 *   tiles_dev, prompt_len_dev, resp_len_dev  int32 [batch]; request b's
 *                    blocks carry prompt_len + resp_len text rows
 *   view_dev         int32 [batch]: the step's view of each request (a level,
 *                    or n_levels for the mixed view)
 *   grid, n_levels, mixed_level, mixed_stride   the view geometry
 *   H, D, scale, out           as for davet_step_attention
 *   cu_seqlens_dev   int32 [batch+1] output, as davet_gather_view writes it
 *   max_total_rows   capacity of out in packed rows
 *   batch            0..256
 * Device-side checks: a view outside [0, n_views) or a negative count sets
 * DAVET_DEV_ARG and the request contributes no rows; a sequence running past
 * store_rows sets DAVET_DEV_ARG (those rows read as zeros); a total above
 * max_total_rows sets DAVET_DEV_CAPACITY and cu_seqlens is clamped.
 */
davet_status davet_view_attention(const void* store, int64_t store_rows, const int64_t* buf_row0_dev,
                                  const int32_t* tiles_dev, const int32_t* prompt_len_dev,
                                  const int32_t* resp_len_dev, const int32_t* view_dev, int batch, int grid,
                                  int n_levels, int mixed_level, int mixed_stride, int H, int D, float scale,
                                  void* out, int32_t* cu_seqlens_dev, int64_t max_total_rows, void* stream);


/* ------------------------------------------------------------ unmasking */

/* Bytes of device workspace that davet_unmask_topk needs for these sizes
 * (batch = number of requests). */
davet_status davet_unmask_topk_workspace(int64_t total_rows, int V, int batch, size_t* bytes);

/*
 * One confidence-ranked commitment step (Sec. 3.1, Eq. 1-2) for a batch of
 * requests.  For every masked answer row i (masked_dev[i] != 0, the set M_t):
 *     argmax_i = smallest w with logits[i][w] = max_w logits[i][w]
 *     conf_i   = 1 / sum_w exp(logits[i][w] - max) (the largest softmax
 *                probability)
 * Then, per request, the min(k, |M_t|) masked rows with the highest conf
 * (ties: lower position first) are committed: tokens_dev[i] = argmax_i and
 * masked_dev[i] = 0; the rest stay masked.  Also returns the inputs of the
 * trajectory risk (Eq. 7): the mean conf over M_t and the churn, the
 * fraction of rows of M_t that had a previous prediction whose argmax
 * changed.
 *   logits        bf16 [total_rows][V]; only masked rows are read.  May be
 *                 device memory or pinned host memory that the device can
 *                 address (cudaHostAlloc / a pinned allocation on a system
 *                 with unified addressing): the kernels then read the masked
 *                 rows over the host link and nothing else crosses it.
 *   V             vocabulary size, a multiple of 8
 *   cu_resp_dev   int32 [batch+1]: request b owns rows cu[b]..cu[b+1]-1;
 *                 cu[batch] <= total_rows
 *   k             commits per request per step, 1..1024
 *   masked_dev    uint8 [total_rows] in/out
 *   tokens_dev    int32 [total_rows] in/out (committed rows written)
 *   argmax_dev    int32 [total_rows] in/out, nullable: in, the previous
 *                 step's argmax (-1 = none); out, this step's argmax for every
 *                 row of M_t.  NULL: churn is reported as 0.
 *   conf_dev      float [total_rows], nullable: conf of every row of M_t
 *   committed_dev int32 [batch][k], nullable: request-local positions
 *                 committed this step in rank order, -1 padded
 *   stats_dev     float [batch][2], nullable: (mean conf over M_t, churn)
 *   workspace     device scratch of davet_unmask_topk_workspace() bytes;
 *                 its contents need no initialization (a call writes every
 *                 entry it reads); calls that may run concurrently need
 *                 separate workspaces
 * Device-side checks: request boundaries outside [0, total_rows] set
 * DAVET_DEV_ARG and are clamped.
 */
davet_status davet_unmask_topk(const void* logits, int V, const int32_t* cu_resp_dev, int batch,
                               int64_t total_rows, int k, uint8_t* masked_dev, int32_t* tokens_dev,
                               int32_t* argmax_dev, float* conf_dev, int32_t* committed_dev, float* stats_dev,
                               void* workspace, size_t workspace_bytes, void* stream);

/* ------------------------------------------------------ allocation policy */

/*
 * Evidence envelope of the denoising-aware allocation policy (Sec. 4.2,
 * Eq. 6), computed once per request before denoising.
 *   T            denoising steps, 1..4096
 *   orientation  0 = early grounding, p_t = 1 - (t - 0.5)/T;
 *                1 = late verification, p_t = (t - 0.5)/T  (t = 1..T)
 *   B, rho       average budget and reserve fraction, in [0, 1]
 *   demand_dev   double [batch] operation demand d(o) in [0, 1] (Table A);
 *                NULL means d = 1 for every request (uniform demand)
 *   lower_dev, upper_dev  double [batch][T] out:
 *                lower = N(p; (1 - rho) B), upper = N(p; (1 - rho + rho d) B),
 *                where N(p; m) = clip(s p, 0, 1) with s >= 0 chosen so that
 *                the mean over the T steps equals m (the normalizer that
 *                rescales the profile and clips it to [0, 1]).
 * Computed in fp64.
 */
davet_status davet_policy_envelope(int T, int orientation, double B, double rho, const double* demand_dev,
                                   int batch, double* lower_dev, double* upper_dev, void* stream);

/*
 * One step of the allocation policy: trajectory risk (Eq. 7), envelope
 * interpolation (Eq. 8) and thirds quantization (Eq. 9), for step t
 * (0-based; the paper's step t+1) of every request.
 *   r = 1 at t = 0; otherwise r = 1 - alpha * cbar * (1 - chi) with
 *   (cbar, chi) = stats_prev_dev[b] from the previous davet_unmask_topk call
 *   (mean confidence over the positions still masked then, and churn);
 *   b_t = lower[t] + r (upper[t] - lower[t]);
 *   view = coarse if b_t < 1/3, mixed if b_t < 2/3, else high.
 *   view_level      host int32 [3]: view index of davet_gather_view used for
 *                   the coarse, mixed and high views (level 0 is the full
 *                   encoding; n_levels is the mixed view)
 *   level_out_dev   int32 [batch] out: the level for davet_gather_view
 *   budget_out_dev  double [batch] out, nullable: b_t
 * Computed in fp64.
 */
davet_status davet_policy_step(int t, int T, const double* lower_dev, const double* upper_dev,
                               const float* stats_prev_dev, int batch, double alpha, const int32_t* view_level,
                               int32_t* level_out_dev, double* budget_out_dev, void* stream);

/*
 * davet_stage_masked_rows -- copies row i (V bf16) of src to row i of dst for
 * every i < total_rows with masked_dev[i] != 0; other rows of dst are left
 * as they are.  The paper has no counterpart: it is input staging for the
 * unmasking (Eq. 2 reads only the still-masked positions' distributions).
 * A caller whose step logits live in pinned host memory can stage step t's
 * rows on a second stream while the GPU runs step t-1, using the mask after
 * step t-2 (a superset of the rows step t reads: commits only clear it), and
 * then call davet_unmask_topk on dst.
 *   src   bf16 [total_rows][V], device-addressable (device memory or pinned
 *         host memory), 16-byte aligned; dst bf16 [total_rows][V] device
 *         memory, 16-byte aligned; V % 8 == 0
 *   masked_dev  uint8 [total_rows]; may change during the call only from
 *         nonzero to zero (a row then copied or not, either is correct for
 *         a later call that reads only rows still masked)
 * One kernel on `stream`.
 */
davet_status davet_stage_masked_rows(const void* src, int V, const uint8_t* masked_dev, int64_t total_rows,
                                     void* dst, void* stream);

/* Size of the scratch array that davet_unmask_topk_noalloc uses (per device). */
#define DAVET_NOALLOC_SCRATCH_BYTES (1u << 20)

/*
 * davet_unmask_topk without a workspace argument.  The paper has no
 * counterpart to this entry point; it exists for callers of this library
 * that cannot allocate device memory of their own.  Examples are plugins that
 * only receive the input and output buffers from a host engine which owns and
 * budgets all device memory, and latency-critical serving loops that must not
 * call cudaMalloc because it can synchronize the device and stall the
 * pipeline.
 *
 * Computes what davet_unmask_topk computes, with the same arguments except
 * the workspace.  Instead of a caller workspace it uses one scratch array of
 * DAVET_NOALLOC_SCRATCH_BYTES (1 MiB) that the library places in device
 * global memory; every device that loads the library holds that array until
 * the process exits.  The call allocates nothing.
 *   - Layout and limit: the scratch holds, per answer row, one 16-byte
 *     (max, sum, first index) record per vocabulary chunk, then a 4-byte
 *     confidence and a 4-byte index; each of these three arrays starts on a
 *     256-byte boundary.  When the chunk count that davet_unmask_topk uses
 *     (16 KB of logits per chunk when the call has at least 8,192 (row,
 *     16 KB chunk) units, else 8 KB; at most 64 chunks) does not fit, this
 *     call cuts each row into fewer, longer chunks until it fits.  The
 *     argmax, the tokens and the committed rows are the same as
 *     davet_unmask_topk's; the confidences and statistics agree to fp32
 *     rounding (the chunk sums are added in a different grouping).  At
 *     V = 126464 the standard layout (31 chunks per row below 512 answer
 *     rows, 16 from 512 on) fits up to 3,970 answer rows.  Only a size that
 *     does not fit even with one chunk per row (24 bytes per row: above
 *     43,680 rows) is rejected, with DAVET_ERR_UNSUPPORTED, before anything
 *     is enqueued.
 *   - Set-up: the array's device address is looked up with
 *     cudaGetSymbolAddress, with the device current, at the first call in
 *     each CUDA context (a device's primary context, or another context the
 *     caller made current) and kept for that context; a context created
 *     later (for example after cudaDeviceReset) gets its own look-up.  Make
 *     the first call in a context before any stream capture.
 *   - Sharing: every call on a device uses the same array, and the array keeps
 *     whatever the last call left in it.  Nothing in it needs clearing: a call
 *     writes every scratch entry it later reads.  Calls whose kernels overlap
 *     on the GPU (for example, issued on two streams with no ordering between
 *     them) race on the array and give wrong results; order them on one
 *     stream or with events.
 */
davet_status davet_unmask_topk_noalloc(const void* logits, int V, const int32_t* cu_resp_dev, int batch,
                                       int64_t total_rows, int k, uint8_t* masked_dev, int32_t* tokens_dev,
                                       int32_t* argmax_dev, float* conf_dev, int32_t* committed_dev,
                                       float* stats_dev, void* stream);

/*
 * Full-layer step (the dense part of one denoising step of the backbone;
 * Sec. 3.1: each step runs the bidirectional transformer over [v_t || q ||
 * y]).  The paper does not print the backbone; the layer here is a
 * pre-normalization decoder layer without a causal mask: RMS normalization,
 * QKV projection with rotary position embedding, davet_step_attention,
 * output projection added to the residual stream, RMS normalization, a
 * gated (SiLU) MLP added to the residual stream; a final normalization of
 * the answer rows and the LM head give the logits davet_unmask_topk reads.
 *
 * davet_linear -- out = epilogue(A . W^T) on the tensor cores (tcgen05,
 * bf16 operands, fp32 accumulation, bf16 output).
 *   A        bf16 [M][K], row-major; W bf16 [N][K], row-major (a linear
 *            layer's weight); K % 64 == 0, N % 256 == 0; 16-byte aligned
 *   out      bf16 [M][N] (epilogue 2: [M][N/2]); must not overlap A or W
 *   epilogue 0 store; 1 out = residual + A.W^T (residual bf16 [M][N], may be
 *            out itself); 2 gated MLP: W holds gate and up rows in alternating
 *            blocks of 128 (rows [256j, 256j+128) gate block j, the next 128
 *            the up block j), out[:, 128j + c] = silu(gate) * up;
 *            3 rotary embedding of columns [0, rope_cols) (query and key
 *            heads of head_dim columns; pairs (d, d + head_dim/2) rotated by
 *            the angle of the row's position in its request, row - cu[b] for
 *            cu_seqlens[b] <= row < cu_seqlens[b+1]), the rest stored as is
 *   cu_seqlens, batch, rope_cols, head_dim (64 or 128), rope_table
 *            (davet_rope_table, [head_dim/2][max_pos] float2), max_pos (the
 *            table's, also its row stride): epilogue 3 only (nullable
 *            otherwise); a position >= max_pos is clamped and flags
 *            DAVET_DEV_ARG
 *   workspace, workspace_bytes   device scratch, nullable.  When the output
 *            tiles would occupy less than half of the SMs (few rows, few
 *            column blocks) and the workspace holds at least
 *            davet_linear_workspace_bytes(M, K, N) bytes (16-byte aligned), K is
 *            split into slices on separate SM pairs whose fp32 partials are
 *            added in slice order (the result does not depend on timing)
 *            before the epilogue; otherwise one pass over K per tile.  A
 *            workspace must not be shared by calls that may run at the same
 *            time.
 *   rows_dev device int32, nullable: the row count to compute, read on the
 *            device when the kernels start (after the previous work on
 *            `stream`), clamped to [0, M] (a count above M flags
 *            DAVET_DEV_CAPACITY, a negative one DAVET_DEV_ARG); rows from
 *            there on are neither read for the epilogue nor written.  M is then the capacity: A, out
 *            and the residual hold M rows, and the tiling and workspace are
 *            chosen for M.  Lets a captured step run a row count that
 *            earlier kernels decide (the allocation policy's views).
 *   row_ss, row_ss_parts, row_ss_eps   nullable: RMS normalization of A's
 *            rows folded into the product.  Row r of A . W^T is multiplied by
 *            1 / sqrt(sum_{j < parts} row_ss[r * parts + j] / K + eps)
 *            before the epilogue (fp32), so that with the normalization gain
 *            folded into W (W[n][k] * gamma[k]) the call computes
 *            rmsnorm(A) . W^T without a normalized copy of A.  row_ss: fp32
 *            [M][parts], partial sums of squares of A's rows (ss_out of the
 *            call that produced A, or davet_row_sumsq).
 *   ss_out   nullable, epilogues 0 and 1 only: fp32 [M][N/256];
 *            ss_out[r * (N/256) + j] = sum of squares of the bf16 values
 *            stored in row r, columns [256j, 256j + 256) (for the next
 *            call's row_ss with parts = N/256).
 * One persistent kernel on `stream` (with a split: a second kernel adds the
 * slices and applies the epilogue).  M > 128 runs on CTA pairs (clusters of
 * two CTAs on two SMs).
 *
 * davet_linear_workspace_bytes -- the workspace davet_linear can use for this
 * shape on the current device (0: none).
 *
 * davet_rope_table -- table[d][p] = (cos, sin)(p * theta^(-2d/head_dim)),
 * fp32, for d < head_dim/2 and p < max_pos (frequency-major, so that rows
 * at consecutive positions read consecutive entries; computed in fp64 on
 * the device).
 *
 * davet_rmsnorm -- out = x / sqrt(mean(x^2) + eps) * gamma per row (fp32
 * sums, bf16 out); x, out bf16 [M][C], gamma bf16 [C], C % 8 == 0.  With
 * cu_resp (int32 [batch+1], the answer-row boundaries) the M = total answer
 * rows are the last cu_resp[b+1] - cu_resp[b] rows of each request's rows
 * (cu_seqlens) and are written packed, in request order.  rows_dev
 * (device int32, nullable): the row count, read on the device and clamped to
 * [0, M], as in davet_linear.
 *
 * davet_row_sumsq -- ss_out[r] = sum over c of x[r][c]^2 (fp32 sums of the
 * bf16 values) for r < M (rows_dev as in davet_linear): row_ss with one part
 * for the first projection of a step.  x bf16 [M][C], C % 8 == 0.
 *
 * davet_embed_answers -- writes the answer rows of the packed step input from
 * an embedding table: row cu_seqlens[b+1] - n_b + i (n_b answer rows of
 * request b) becomes table[tokens[cu_resp[b] + i]], or table[mask_id] while
 * the token is still masked (< 0); a token >= V uses mask_id and flags
 * DAVET_DEV_ARG.  table bf16 [V][C]; x bf16 [rows][C].
 */
davet_status davet_linear(const void* A, int64_t M, int K, const void* W, int N, void* out, int epilogue,
                          const void* residual, const int32_t* cu_seqlens, int batch, int rope_cols, int head_dim,
                          const void* rope_table, int max_pos, void* workspace, size_t workspace_bytes,
                          const float* row_ss, int row_ss_parts, float row_ss_eps, float* ss_out,
                          const int32_t* rows_dev, void* stream);
davet_status davet_linear_workspace_bytes(int64_t M, int K, int N, size_t* bytes);
davet_status davet_rope_table(int max_pos, int head_dim, double theta, void* table, void* stream);
davet_status davet_rmsnorm(const void* x, int64_t M, int C, const void* gamma, float eps, void* out,
                           const int32_t* cu_seqlens, const int32_t* cu_resp, int batch, const int32_t* rows_dev,
                           void* stream);
davet_status davet_row_sumsq(const void* x, int64_t M, int C, float* ss_out, const int32_t* rows_dev, void* stream);
davet_status davet_embed_answers(const void* table, int V, int C, const int32_t* tokens, int mask_id,
                                 const int32_t* cu_seqlens, const int32_t* cu_resp, int batch, int64_t total_resp,
                                 void* x, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* DAVET_H_ */
