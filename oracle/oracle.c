/*
 * oracle.c -- plain fp64 CPU definitions of the DAVET step-conditioning path.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may link, load or
 * call this file; only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg use it.  It shares no code, header, table or helper with
 * the CUDA library.
 *
 * Every routine is the plain definition of what the step computes, written
 * with straightforward loops in double precision so that it can be checked
 * against the paper by eye:
 *
 *   oracle_pyramid_*     Sec. 4.3: the evidence realizer builds an ordered
 *                        hierarchy of views from one visual encoding by
 *                        structured pooling; level 0 is the unpooled view
 *                        (v^(K) = v).  Reading: 2x2 stride-2 cascade, each
 *                        output the mean of its in-range children.
 *   oracle_gather        Sec. 3.2 / Eq. 5: the step input is the chosen view
 *                        followed by the query and the answer state.
 *   oracle_attention_*   Sec. 3.1 / Eq. 1: bidirectional (non-causal)
 *                        attention over the whole packed sequence.
 *   oracle_softmax_row,  Sec. 3.1 / Eq. 1-2: per masked position the token
 *   oracle_unmask        distribution, its argmax, and the confidence-ranked
 *                        commitment of the top-k positions; Sec. 4.2 / Eq. 7
 *                        defines the mean confidence and churn statistics.
 *   oracle_mixed_view    Sec. 4.3: the `mixed` view, coarse pooled tokens plus
 *                        a fixed subset of unpooled tokens (a centred lattice).
 *   oracle_policy_*      Sec. 4.2 / Eq. 6-8 and Sec. 4.3 / Eq. 9: phase
 *                        profile, normalizer, evidence envelope, trajectory
 *                        risk, envelope interpolation, thirds quantization.
 *   oracle_prune_keep    Sec. 4.3 / Sec. 5.3: nested visual-token pruning,
 *                        the kept tokens of every view for a given score.
 *   oracle_merge_views   Sec. 4.3 / Sec. 5.3: hierarchical similarity merging
 *                        (bipartite matching rounds level by level).  Its
 *                        merge decisions are taken in binary32 with a fixed
 *                        operation order (fused multiply-add chains in
 *                        ascending channel order, correctly rounded square
 *                        root and division), the precision the CUDA kernels
 *                        decide in, so both sides take the same decisions;
 *                        the file is compiled without contraction of
 *                        separate multiplies and adds.
 *
 * Parallelism: OpenMP over independent outer loops only (tiles, requests x
 * heads, rows); each inner computation is the sequential definition.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* ---------------------------------------------------------------- helpers */

/* bf16 is the upper half of an IEEE binary32; widening to double is exact. */
static double bf16_to_f64(uint16_t h)
{
    uint32_t u = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

int oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* ---------------------------------------------------------------- pyramid */

/* Side of every level: G_0 = grid, G_l = ceil(G_{l-1} / 2). Returns the
 * number of rows one tile contributes to all levels together. */
int64_t oracle_level_sides(int grid, int n_levels, int *side)
{
    int64_t rows = 0;
    int g = grid;
    for (int l = 0; l < n_levels; ++l) {
        side[l] = g;
        rows += (int64_t)g * g;
        g = (g + 1) / 2;
    }
    return rows;
}

/*
 * Pyramid over n_tiles independent grid x grid tiles of C channels.
 * in : feat[t][y][x][c]                      (level 0 itself)
 * out: level-major, tile-major within a level:
 *      row(l, t, y, x) = off_l + t*G_l^2 + y*G_l + x,
 *      off_l = n_tiles * sum_{j<l} G_j^2,    out[row*C + c].
 * Level l cell (y,x) is the mean of the level l-1 cells (2y+i, 2x+j),
 * i,j in {0,1}, that lie inside the level l-1 grid.
 */
void oracle_pyramid_f64(const double *feat, int n_tiles, int grid, int n_levels,
                        int C, double *out)
{
    int side[32];
    oracle_level_sides(grid, n_levels, side);
    int64_t off[33];
    off[0] = 0;
    for (int l = 0; l < n_levels; ++l)
        off[l + 1] = off[l] + (int64_t)n_tiles * side[l] * side[l];

    /* level 0: the unpooled view */
    for (int64_t i = 0; i < (int64_t)n_tiles * grid * grid * C; ++i)
        out[i] = feat[i];

    for (int l = 1; l < n_levels; ++l) {
        const int gp = side[l - 1], g = side[l];
#pragma omp parallel for schedule(static)
        for (int t = 0; t < n_tiles; ++t) {
            for (int y = 0; y < g; ++y) {
                for (int x = 0; x < g; ++x) {
                    double *dst = out + (off[l] + (int64_t)t * g * g + (int64_t)y * g + x) * C;
                    for (int c = 0; c < C; ++c) {
                        double sum = 0.0;
                        int count = 0;
                        for (int i = 0; i < 2; ++i) {
                            for (int j = 0; j < 2; ++j) {
                                const int yy = 2 * y + i, xx = 2 * x + j;
                                if (yy < gp && xx < gp) {
                                    const int64_t src = off[l - 1] + (int64_t)t * gp * gp
                                                      + (int64_t)yy * gp + xx;
                                    sum += out[src * C + c];
                                    count += 1;
                                }
                            }
                        }
                        dst[c] = sum / count;
                    }
                }
            }
        }
    }
}

/* Same pyramid with bf16 input; the inputs are widened exactly. */
void oracle_pyramid_bf16(const uint16_t *feat, int n_tiles, int grid, int n_levels,
                         int C, double *out)
{
    const int64_t n = (int64_t)n_tiles * grid * grid * C;
    double *wide = (double *)malloc((size_t)n * sizeof(double));
    if (!wide) return;
    for (int64_t i = 0; i < n; ++i) wide[i] = bf16_to_f64(feat[i]);
    oracle_pyramid_f64(wide, n_tiles, grid, n_levels, C, out);
    free(wide);
}

/* ----------------------------------------------------------------- gather */

/*
 * Packs, for every request b, the rows of its view at level level[b]
 * (all tiles of that level in tile order, row-major within a tile) followed
 * by its P_b prompt rows and R_b response rows taken from
 * text[text_off[b] ...].  Rows are C bf16 values and are copied bit for bit.
 * pyr[b] is request b's pyramid in the layout of oracle_pyramid_f64; when
 * mixed_rows_per_tile > 0, its mixed view (oracle_mixed_view) follows the
 * pooled levels and level index n_levels selects it.
 * cu[b] is the first packed row of request b; cu[batch] the total.
 */
void oracle_gather_mixed(const uint16_t *const *pyr, const int32_t *tiles,
                         const uint16_t *text, const int64_t *text_off,
                         const int32_t *prompt_len, const int32_t *resp_len,
                         const int32_t *level, int batch, int grid, int n_levels, int C,
                         int mixed_rows_per_tile, uint16_t *out, int32_t *cu)
{
    int side[32];
    oracle_level_sides(grid, n_levels, side);
    int64_t row = 0;
    cu[0] = 0;
    for (int b = 0; b < batch; ++b) {
        const int l = level[b];
        /* level index n_levels names the mixed view, stored after the pooled levels */
        int64_t level_start = 0;
        for (int j = 0; j < l && j < n_levels; ++j) level_start += (int64_t)tiles[b] * side[j] * side[j];
        const int64_t n_vis = l < n_levels ? (int64_t)tiles[b] * side[l] * side[l]
                                           : (int64_t)tiles[b] * mixed_rows_per_tile;
        for (int64_t r = 0; r < n_vis; ++r, ++row)
            memcpy(out + row * C, pyr[b] + (level_start + r) * C, (size_t)C * 2);
        const int64_t n_text = (int64_t)prompt_len[b] + resp_len[b];
        for (int64_t r = 0; r < n_text; ++r, ++row)
            memcpy(out + row * C, text + (text_off[b] + r) * C, (size_t)C * 2);
        cu[b + 1] = (int32_t)row;
    }
}

void oracle_gather(const uint16_t *const *pyr, const int32_t *tiles,
                   const uint16_t *text, const int64_t *text_off,
                   const int32_t *prompt_len, const int32_t *resp_len,
                   const int32_t *level, int batch, int grid, int n_levels, int C,
                   uint16_t *out, int32_t *cu)
{
    oracle_gather_mixed(pyr, tiles, text, text_off, prompt_len, resp_len, level, batch, grid, n_levels, C,
                        0, out, cu);
}

/* -------------------------------------------------------------- attention */

/* qkv[n][s][h][d], s = 0 (query), 1 (key), 2 (value). */
static double qkv_at(const uint16_t *qkv, int64_t n, int s, int h, int d, int H, int D)
{
    return bf16_to_f64(qkv[((n * 3 + s) * (int64_t)H + h) * D + d]);
}

/*
 * Output row `row`, head h: o = sum_j softmax_j(scale * q . k_j) v_j over
 * all key rows j of the same request (no causal mask).  The row maximum is
 * subtracted before exponentiating, which leaves the result unchanged.
 */
static void attention_one(const uint16_t *qkv, int64_t start, int64_t end, int64_t row,
                          int h, int H, int D, double scale, double *o, double *w)
{
    double m = -INFINITY;
    for (int64_t j = start; j < end; ++j) {
        double s = 0.0;
        for (int d = 0; d < D; ++d)
            s += qkv_at(qkv, row, 0, h, d, H, D) * qkv_at(qkv, j, 1, h, d, H, D);
        s *= scale;
        w[j - start] = s;
        if (s > m) m = s;
    }
    double denom = 0.0;
    for (int64_t j = start; j < end; ++j) {
        w[j - start] = exp(w[j - start] - m);
        denom += w[j - start];
    }
    for (int d = 0; d < D; ++d) o[d] = 0.0;
    for (int64_t j = start; j < end; ++j)
        for (int d = 0; d < D; ++d)
            o[d] += w[j - start] * qkv_at(qkv, j, 2, h, d, H, D);
    for (int d = 0; d < D; ++d) o[d] /= denom;
}

/* Dense attention for every row and head; out[n][h][d]. */
void oracle_attention(const uint16_t *qkv, const int32_t *cu, int batch, int H, int D,
                      double scale, double *out)
{
    for (int b = 0; b < batch; ++b) {
        const int64_t start = cu[b], end = cu[b + 1];
        const int64_t L = end - start;
        if (L <= 0) continue;
#pragma omp parallel
        {
            double *w = (double *)malloc((size_t)L * sizeof(double));
#pragma omp for schedule(dynamic, 1) collapse(2)
            for (int h = 0; h < H; ++h)
                for (int64_t i = start; i < end; ++i)
                    attention_one(qkv, start, end, i, h, H, D, scale,
                                  out + (i * H + h) * D, w);
            free(w);
        }
    }
}

/*
 * The same definition evaluated only at n_items sampled (row, head) pairs;
 * out[item][d].  The request of each row is found from cu.
 */
void oracle_attention_rows(const uint16_t *qkv, const int32_t *cu, int batch, int H, int D,
                           double scale, int64_t n_items, const int64_t *rows,
                           const int32_t *heads, double *out)
{
    int64_t max_len = 0;
    for (int b = 0; b < batch; ++b)
        if (cu[b + 1] - cu[b] > max_len) max_len = cu[b + 1] - cu[b];
#pragma omp parallel
    {
        double *w = (double *)malloc((size_t)(max_len > 0 ? max_len : 1) * sizeof(double));
#pragma omp for schedule(dynamic, 1)
        for (int64_t it = 0; it < n_items; ++it) {
            const int64_t r = rows[it];
            int b = 0;
            while (b < batch && !(r >= cu[b] && r < cu[b + 1])) ++b;
            if (b == batch) continue;
            attention_one(qkv, cu[b], cu[b + 1], r, heads[it], H, D, scale, out + it * D, w);
        }
        free(w);
    }
}

/* -------------------------------------------------------------- unmasking */

/* p_w = exp(l_w - max) / sum_v exp(l_v - max) for one row of V logits. */
void oracle_softmax_row(const uint16_t *logits, int V, double *p)
{
    double m = -INFINITY;
    for (int w = 0; w < V; ++w) {
        const double l = bf16_to_f64(logits[w]);
        if (l > m) m = l;
    }
    double denom = 0.0;
    for (int w = 0; w < V; ++w) {
        p[w] = exp(bf16_to_f64(logits[w]) - m);
        denom += p[w];
    }
    for (int w = 0; w < V; ++w) p[w] /= denom;
}

/* argmax with ties resolved to the lowest vocabulary index */
static int argmax_first(const uint16_t *logits, int V)
{
    int best = 0;
    double m = bf16_to_f64(logits[0]);
    for (int w = 1; w < V; ++w) {
        const double l = bf16_to_f64(logits[w]);
        if (l > m) { m = l; best = w; }
    }
    return best;
}

typedef struct { double conf; int32_t pos; } ranked_t;

/* order: higher confidence first, then lower position */
static int ranked_cmp(const void *a, const void *b)
{
    const ranked_t *x = (const ranked_t *)a, *y = (const ranked_t *)b;
    if (x->conf > y->conf) return -1;
    if (x->conf < y->conf) return 1;
    return (x->pos > y->pos) - (x->pos < y->pos);
}

/*
 * One confidence-ranked commitment step (Eq. 1-2).
 *   logits[row][V]   rows = answer positions of all requests; request b owns
 *                    rows cu_resp[b] .. cu_resp[b+1]-1; only masked rows are
 *                    read.
 *   masked[row]      in: 1 for positions in M_t; out: committed rows set to 0.
 *   tokens[row]      committed rows receive their argmax token.
 *   argmax[row]      in: the previous step's argmax (-1 = none); out: this
 *                    step's argmax for every row of M_t.
 *   conf[row]        out for rows of M_t: the max softmax probability.
 *   committed[b][k]  out: request-local positions committed this step, in
 *                    rank order, -1 padded.
 *   stats[b][2]      out: mean confidence over M_t, and churn = the fraction
 *                    of rows of M_t that also had a previous prediction whose
 *                    argmax changed (0 when no row had one).
 */
void oracle_unmask(const uint16_t *logits, int V, const int32_t *cu_resp, int batch, int k,
                   uint8_t *masked, int32_t *tokens, int32_t *argmax, double *conf,
                   int32_t *committed, double *stats)
{
    const int64_t n_rows = cu_resp[batch];

    /* confidence of every masked row: softmax probability of its argmax */
#pragma omp parallel
    {
        double *pr = (double *)malloc((size_t)V * sizeof(double));
#pragma omp for schedule(dynamic, 4)
        for (int64_t i = 0; i < n_rows; ++i) {
            if (!masked[i]) continue;
            const uint16_t *row = logits + i * (int64_t)V;
            oracle_softmax_row(row, V, pr);
            conf[i] = pr[argmax_first(row, V)];
        }
        free(pr);
    }

    for (int b = 0; b < batch; ++b) {
        const int64_t s = cu_resp[b], e = cu_resp[b + 1];
        int64_t n_masked = 0, n_both = 0, n_changed = 0;
        double conf_sum = 0.0;
        ranked_t *cand = (ranked_t *)malloc((size_t)((e - s) > 0 ? (e - s) : 1) * sizeof(ranked_t));
        for (int64_t i = s; i < e; ++i) {
            if (!masked[i]) continue;
            const int a = argmax_first(logits + i * (int64_t)V, V);
            if (argmax[i] >= 0) {
                n_both += 1;
                if (argmax[i] != a) n_changed += 1;
            }
            argmax[i] = a;
            conf_sum += conf[i];
            cand[n_masked].conf = conf[i];
            cand[n_masked].pos = (int32_t)(i - s);
            n_masked += 1;
        }
        qsort(cand, (size_t)n_masked, sizeof(ranked_t), ranked_cmp);
        const int64_t take = n_masked < k ? n_masked : k;
        for (int j = 0; j < k; ++j) committed[(int64_t)b * k + j] = -1;
        for (int64_t j = 0; j < take; ++j) {
            const int64_t i = s + cand[j].pos;
            tokens[i] = argmax[i];
            masked[i] = 0;
            committed[(int64_t)b * k + j] = cand[j].pos;
        }
        stats[2 * b + 0] = n_masked ? conf_sum / (double)n_masked : 0.0;
        stats[2 * b + 1] = n_both ? (double)n_changed / (double)n_both : 0.0;
        free(cand);
    }
}

/* ----------------------------------------------------------------- policy */

/*
 * Phase profile of Sec. 4.2: p_t = 1 - (t - 0.5)/T (early grounding,
 * orientation 0) or p_t = (t - 0.5)/T (late verification, orientation 1),
 * for t = 1..T; p[t-1] holds p_t.
 */
void oracle_policy_profile(int T, int orientation, double *p)
{
    for (int t = 1; t <= T; ++t) {
        const double u = (t - 0.5) / (double)T;
        p[t - 1] = orientation == 0 ? 1.0 - u : u;
    }
}

static double mean_clipped(const double *p, int T, double s)
{
    double acc = 0.0;
    for (int t = 0; t < T; ++t) {
        double v = s * p[t];
        if (v < 0.0) v = 0.0;
        if (v > 1.0) v = 1.0;
        acc += v;
    }
    return acc / T;
}

/*
 * Normalizer N(p; target) of Sec. 4.2: rescale the profile and clip it to
 * [0,1] so that its mean equals the target.  Reading: a multiplicative scale
 * s >= 0, out_t = clip(s * p_t, 0, 1), with s found by bisection on the
 * mean, which is continuous and non-decreasing in s.  Targets at or above
 * the largest reachable mean give all ones; targets <= 0 give all zeros.
 */
void oracle_policy_normalize(const double *p, int T, double target, double *out)
{
    double pmin = INFINITY, pmax = 0.0;
    for (int t = 0; t < T; ++t) {
        if (p[t] > 0.0 && p[t] < pmin) pmin = p[t];
        if (p[t] > pmax) pmax = p[t];
    }
    double lo = 0.0, hi = (pmin < INFINITY) ? 1.0 / pmin : 0.0;
    if (target <= 0.0 || pmax <= 0.0) {
        hi = 0.0;
    } else if (mean_clipped(p, T, hi) <= target) {
        lo = hi;
    } else {
        for (int it = 0; it < 200; ++it) {
            const double mid = 0.5 * (lo + hi);
            if (mean_clipped(p, T, mid) < target) lo = mid; else hi = mid;
        }
    }
    const double s = (target <= 0.0 || pmax <= 0.0) ? 0.0 : 0.5 * (lo + hi);
    for (int t = 0; t < T; ++t) {
        double v = s * p[t];
        if (v < 0.0) v = 0.0;
        if (v > 1.0) v = 1.0;
        out[t] = v;
    }
}

/* Evidence envelope, Eq. 6: lower = N(p; (1-rho)B), upper = N(p; (1-rho+rho d)B). */
void oracle_policy_envelope(const double *p, int T, double B, double rho, double demand,
                            double *lower, double *upper)
{
    oracle_policy_normalize(p, T, (1.0 - rho) * B, lower);
    oracle_policy_normalize(p, T, (1.0 - rho + rho * demand) * B, upper);
}

/* Trajectory risk, Eq. 7: r_1 = 1; r_t = 1 - alpha * cbar_{t-1} * (1 - chi_{t-1}). */
double oracle_policy_risk(int t, double alpha, double cbar_prev, double chi_prev)
{
    if (t <= 1) return 1.0;
    return 1.0 - alpha * cbar_prev * (1.0 - chi_prev);
}

/* Envelope interpolation, Eq. 8. */
double oracle_policy_budget(double lower_t, double upper_t, double r_t)
{
    return lower_t + r_t * (upper_t - lower_t);
}

/* Thirds quantization, Eq. 9: 0 = coarse (b < 1/3), 1 = mixed, 2 = high (b >= 2/3). */
int oracle_policy_view(double b)
{
    if (b < 1.0 / 3.0) return 0;
    if (b < 2.0 / 3.0) return 1;
    return 2;
}

/* ------------------------------------------------------------- mixed view */

/*
 * The `mixed` evidence view of Sec. 4.3: the pooled (`coarse`) representation
 * augmented with a fixed subset of unpooled tokens.  Reading: per tile, all
 * rows of pyramid level `coarse_level` (row-major), followed by the level-0
 * tokens on a centred stride-`stride` lattice, (y, x) with
 * y = stride/2 + i*stride < grid and x = stride/2 + j*stride < grid, row-major;
 * tiles follow one another.  `pyr` is a level-major pyramid of n_tiles tiles
 * (layout of oracle_pyramid_f64) holding bf16 bits; rows are copied bit for
 * bit.  Returns the rows written (rows per tile times n_tiles).
 */
int64_t oracle_mixed_view(const uint16_t *pyr, int n_tiles, int grid, int n_levels, int coarse_level,
                          int stride, int C, uint16_t *out)
{
    int side[32];
    oracle_level_sides(grid, n_levels, side);
    int64_t off[33];
    off[0] = 0;
    for (int l = 0; l < n_levels; ++l)
        off[l + 1] = off[l] + (int64_t)n_tiles * side[l] * side[l];
    const int gc = side[coarse_level];
    int64_t row = 0;
    for (int t = 0; t < n_tiles; ++t) {
        for (int i = 0; i < gc * gc; ++i, ++row)
            memcpy(out + row * C, pyr + (off[coarse_level] + (int64_t)t * gc * gc + i) * C, (size_t)C * 2);
        for (int y = stride / 2; y < grid; y += stride)
            for (int x = stride / 2; x < grid; x += stride, ++row)
                memcpy(out + row * C, pyr + ((int64_t)t * grid * grid + (int64_t)y * grid + x) * C, (size_t)C * 2);
    }
    return row;
}

/* ------------------------------------------------------ pruning realizer */

/*
 * Order key of an importance score: larger scores first, a NaN below every
 * number, equal scores by ascending token index (the sort is then total).
 */
typedef struct {
    float s;
    int32_t i;
} scored_t;

static int scored_cmp(const void *a, const void *b)
{
    const scored_t *x = (const scored_t *)a, *y = (const scored_t *)b;
    const int xn = isnan(x->s), yn = isnan(y->s);
    if (xn != yn) return xn ? 1 : -1;
    if (!xn && x->s != y->s) return x->s > y->s ? -1 : 1;
    return x->i < y->i ? -1 : (x->i > y->i);
}

/*
 * Nested visual-token pruning (Sec. 4.3 "compatible evidence realizers":
 * pruning varies the retention ratio; Sec. 5.3 / Table 2).  The importance
 * score is not specified by the paper and is an input here: score[t][i] for
 * token i (raster order) of tile t.  Reading: view v keeps, per tile, the
 * rows_per_tile[v] highest-scoring tokens (ties by smaller index, NaN last)
 * in raster order, so each view is a subset of every larger one.
 * keep: the kept token indices, view-major then tile-major,
 *       keep[sum_{u<v} n_tiles*m_u + t*m_v + j]  (m_v = rows_per_tile[v]).
 */
void oracle_prune_keep(const float *score, int n_tiles, int grid, int n_views, const int32_t *rows_per_tile,
                       int32_t *keep)
{
    const int n = grid * grid;
    int64_t base[33];
    base[0] = 0;
    for (int v = 0; v < n_views; ++v) base[v + 1] = base[v] + (int64_t)n_tiles * rows_per_tile[v];
#pragma omp parallel for schedule(dynamic)
    for (int t = 0; t < n_tiles; ++t) {
        scored_t *s = malloc(sizeof(scored_t) * (size_t)n);
        int32_t *rank = malloc(sizeof(int32_t) * (size_t)n);
        for (int i = 0; i < n; ++i) {
            s[i].s = score[(int64_t)t * n + i];
            s[i].i = i;
        }
        qsort(s, (size_t)n, sizeof *s, scored_cmp);
        for (int p = 0; p < n; ++p) rank[s[p].i] = p;
        for (int v = 0; v < n_views; ++v) {
            int32_t *k = keep + base[v] + (int64_t)t * rows_per_tile[v];
            int j = 0;
            for (int i = 0; i < n; ++i)
                if (rank[i] < rows_per_tile[v]) k[j++] = i;
        }
        free(rank);
        free(s);
    }
}

/* ------------------------------------------------------ merging realizer */

static float bf16_to_f32(uint16_t h)
{
    uint32_t u = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return f;
}

/* binary32 -> bfloat16, round to nearest, ties to even (finite inputs). */
static uint16_t f32_to_bf16_rne(float f)
{
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    if ((u & 0x7f800000u) == 0x7f800000u) return (uint16_t)((u >> 16) | ((u & 0xffffu) ? 0x40u : 0u));
    u += 0x7fffu + ((u >> 16) & 1u);
    return (uint16_t)(u >> 16);
}

/*
 * Feature sums of the current tokens: S[j][c] = sum over the level-0 tokens
 * i with tok[i] == j, in ascending i, of x_i[c0 + c] (binary32, one rounded
 * addition per member, starting from the first member's value).
 */
static void member_sums(const uint16_t *x0, int n0, const int32_t *tok, int n, int C, int c0, int Cs, float *S,
                        int32_t *size)
{
    for (int j = 0; j < n; ++j) size[j] = 0;
    for (int i = 0; i < n0; ++i) {
        const int j = tok[i];
        float *s = S + (int64_t)j * Cs;
        const uint16_t *x = x0 + (int64_t)i * C + c0;
        if (size[j] == 0)
            for (int c = 0; c < Cs; ++c) s[c] = bf16_to_f32(x[c]);
        else
            for (int c = 0; c < Cs; ++c) s[c] = s[c] + bf16_to_f32(x[c]);
        ++size[j];
    }
}

/* Inverse norm 1/sqrt(sum_c s_c^2) with the squares accumulated by fused
 * multiply-adds in ascending c; a zero vector gets 0. */
static float inv_norm(const float *s, int Cs)
{
    float n2 = 0.0f;
    for (int c = 0; c < Cs; ++c) n2 = fmaf(s[c], s[c], n2);
    return n2 > 0.0f ? 1.0f / sqrtf(n2) : 0.0f;
}

/*
 * One bipartite matching round over the n current tokens of one tile
 * (token merging by bipartite soft matching, Bolya et al. 2023, as the
 * aggregation step).  Positions 0, 2, 4, ... form set A and 1, 3, 5, ... set
 * B.  Each a in A is matched to the b in B of highest cosine similarity
 *   sim(a, b) = (dot(S_a, S_b) * inv_a) * inv_b,
 * dot accumulated by fused multiply-adds in ascending channel order (ties
 * go to the smaller b).  The r members of A with the highest matched
 * similarity (ties to the smaller position) are merged into their match; the
 * survivors keep their relative order.  Updates tok and returns n - r.
 */
static int merge_round(const uint16_t *x0, int n0, int32_t *tok, int n, int r, int C, int c0, int Cs, float *S,
                       int32_t *size, float *inv, float *best, int32_t *best_b, int32_t *newpos)
{
    member_sums(x0, n0, tok, n, C, c0, Cs, S, size);
    for (int j = 0; j < n; ++j) inv[j] = inv_norm(S + (int64_t)j * Cs, Cs);
    const int nA = (n + 1) / 2, nB = n / 2;
    for (int a = 0; a < nA; ++a) {
        const float *sa = S + (int64_t)(2 * a) * Cs;
        best[a] = 0.0f;
        best_b[a] = -1;
        for (int b = 0; b < nB; ++b) {
            const float *sb = S + (int64_t)(2 * b + 1) * Cs;
            float dot = 0.0f;
            for (int c = 0; c < Cs; ++c) dot = fmaf(sa[c], sb[c], dot);
            const float sim = (dot * inv[2 * a]) * inv[2 * b + 1];
            if (best_b[a] < 0 || sim > best[a]) {
                best[a] = sim;
                best_b[a] = b;
            }
        }
    }
    /* merged[a] <=> fewer than r members of A rank before a */
    int32_t *merged = newpos + n; /* scratch of nA entries after newpos */
    for (int a = 0; a < nA; ++a) {
        int before = 0;
        for (int o = 0; o < nA; ++o)
            if (best[o] > best[a] || (best[o] == best[a] && o < a)) ++before;
        merged[a] = before < r;
    }
    int kept = 0;
    for (int p = 0; p < n; ++p) {
        const int gone = (p % 2 == 0) && merged[p / 2];
        newpos[p] = gone ? -1 : kept++;
    }
    for (int i = 0; i < n0; ++i) {
        int p = tok[i];
        if (p % 2 == 0 && merged[p / 2]) p = 2 * best_b[p / 2] + 1;
        tok[i] = newpos[p];
    }
    return kept;
}

/* One matching round of one tile on its own (for the tests): tok is
 * updated in place; best / best_b (nullable, ceil(n/2) entries) receive each
 * member of A's matched similarity and B index.  Returns the new count. */
int oracle_merge_round(const uint16_t *x0, int n0, int C, int c0, int Cs, int32_t *tok, int n, int r, float *best,
                       int32_t *best_b)
{
    float *S = malloc(sizeof(float) * (size_t)n * (size_t)Cs);
    int32_t *size = malloc(sizeof(int32_t) * (size_t)n);
    float *inv = malloc(sizeof(float) * (size_t)n);
    float *bs = malloc(sizeof(float) * (size_t)n);
    int32_t *bb = malloc(sizeof(int32_t) * (size_t)n);
    int32_t *newpos = malloc(sizeof(int32_t) * (size_t)(2 * n));
    const int out = merge_round(x0, n0, tok, n, r, C, c0, Cs, S, size, inv, bs, bb, newpos);
    for (int a = 0; a < (n + 1) / 2; ++a) {
        if (best) best[a] = bs[a];
        if (best_b) best_b[a] = bb[a];
    }
    free(newpos);
    free(bb);
    free(bs);
    free(inv);
    free(size);
    free(S);
    return out;
}

/*
 * Hierarchical similarity merging (Sec. 4.3 "compatible evidence realizers":
 * merging varies the aggregation strength; Sec. 5.3 / Table 2).  Reading:
 * per tile, level 0 is the encoding; level l is built from level l-1 by
 * bipartite matching rounds (merge_round) with r = min(n - G_l^2, ceil(n/2))
 * until it holds G_l^2 tokens, the row count of the pooled level l, so the
 * views have the pooled hierarchy's lengths.  Similarity is measured on
 * channels [c0, c0 + Cs) of the token sums.  A merged token's row is the
 * mean of the level-0 rows it absorbed: the binary32 sum of its members in
 * ascending index, divided by their count (binary32 division), rounded to
 * bf16 (nearest even).
 * feat : bf16 bits [n_tiles][grid*grid][C]
 * out  : bf16 bits, level-major then tile-major, levels 1..n_levels-1:
 *        row(l, t, j) = sum_{1<=u<l} n_tiles*G_u^2 + t*G_l^2 + j
 * assign (nullable): int32 [n_levels][n_tiles][grid*grid], the level-l token
 *        index that level-0 token i belongs to (level 0: i itself)
 */
void oracle_merge_views(const uint16_t *feat, int n_tiles, int grid, int n_levels, int C, int c0, int Cs,
                        uint16_t *out, int32_t *assign)
{
    int side[32];
    oracle_level_sides(grid, n_levels, side);
    const int n0 = grid * grid;
    int64_t lbase[33];
    lbase[1] = 0;
    for (int l = 1; l < n_levels; ++l) lbase[l + 1] = lbase[l] + (int64_t)n_tiles * side[l] * side[l];
#pragma omp parallel for schedule(dynamic)
    for (int t = 0; t < n_tiles; ++t) {
        const uint16_t *x0 = feat + (int64_t)t * n0 * C;
        int32_t *tok = malloc(sizeof(int32_t) * (size_t)n0);
        float *S = malloc(sizeof(float) * (size_t)n0 * (size_t)(Cs > C ? Cs : C));
        int32_t *size = malloc(sizeof(int32_t) * (size_t)n0);
        float *inv = malloc(sizeof(float) * (size_t)n0);
        float *best = malloc(sizeof(float) * (size_t)n0);
        int32_t *best_b = malloc(sizeof(int32_t) * (size_t)n0);
        int32_t *newpos = malloc(sizeof(int32_t) * (size_t)(2 * n0));
        for (int i = 0; i < n0; ++i) tok[i] = i;
        if (assign)
            for (int i = 0; i < n0; ++i) assign[(int64_t)t * n0 + i] = i;
        int n = n0;
        for (int l = 1; l < n_levels; ++l) {
            const int target = side[l] * side[l];
            while (n > target) {
                const int nA = (n + 1) / 2;
                const int r = n - target < nA ? n - target : nA;
                n = merge_round(x0, n0, tok, n, r, C, c0, Cs, S, size, inv, best, best_b, newpos);
            }
            member_sums(x0, n0, tok, n, C, 0, C, S, size);
            for (int j = 0; j < n; ++j)
                for (int c = 0; c < C; ++c)
                    out[(lbase[l] + (int64_t)t * target + j) * C + c] =
                        f32_to_bf16_rne(S[(int64_t)j * C + c] / (float)size[j]);
            if (assign)
                for (int i = 0; i < n0; ++i) assign[((int64_t)l * n_tiles + t) * n0 + i] = tok[i];
        }
        free(newpos);
        free(best_b);
        free(best);
        free(inv);
        free(size);
        free(S);
        free(tok);
    }
}
