/*
 * dge_oracle.c -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously correct float64 CPU restatement of the
 * Draft-Guided Eviction score -> select -> compact pass.  It exists to check
 * the CUDA path; nothing in the product links it.  Only tests/, the smoke
 * check and bench.py's CPU-baseline leg may load it.  It shares no code,
 * header, table or constant with the CUDA library.
 *
 * Every input is the exact bf16 value widened to double; all arithmetic is
 * double.  No blocking, fusion or reordering beyond the definitions below.
 *
 * Passages followed (paper sections / equations / algorithms):
 *   - Alg. 1 line B: s = sum over observation queries of
 *     softmax(q K^T / sqrt(d)); the DGE-W alternative scores the window rows.
 *   - App. B: float32 softmax over the observation rows, score summed over
 *     past keys, max-pool kernel 7, per-head top-B.
 *   - App. G ("Removing it, measured"): scores aggregated over the query heads
 *     of one KV group (sum here; a positive factor does not change ranking).
 *   - App. E implementation notes: sort kept indices to keep temporal order,
 *     gather [retained past] || [window + draft tail].
 *   - Table "complexity", note a: H2O accumulates softmax attention over all
 *     prompt rows (and the draft rows); causal.
 *   - App. L, composition: StreamingLLM keeps 4 sinks plus a recency window.
 *   - App. L, PyramidKV's discrete schedule: c = B - w, min = floor(c/20),
 *     max = 2c - min, steps = floor((max - min)/(L - 1)), budget_l = max - l*steps.
 *
 * Readings where the paper is silent (see the design notes of the repo):
 *   causal visibility (row at position p sees keys j <= p), sum over rows and
 *   group heads, pooling over the past range only (max ignores out-of-range
 *   cells, avg divides by the full kernel with zero padding), ties broken by
 *   the lower position, every budget counts every protected position.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define DGEO_POOL_NONE 0
#define DGEO_POOL_MAX 1
#define DGEO_POOL_AVG 2

static double bf16_value(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/*
 * Attention scores of one KV head (Alg. 1 line B; App. B; App. G).
 *
 *   Q      [R][d] bf16 bits: the observation rows of the G query heads of the
 *          group, stacked; row r sits at cache position pos[r].
 *   K      [n][d] bf16 bits.
 *   scale  logit scale (1/sqrt(d) in the paper).
 *   P      number of scored positions [0, P).
 *   raw    out [P]: raw[j] = sum_r exp(s_rj - lse_r) over rows with j <= pos[r].
 *   lse    out [R] (may be NULL): lse_r = log sum_{j <= pos[r]} exp(s_rj).
 *   work   scratch of n doubles.
 */
static void scores_unit(const uint16_t *Q, const uint16_t *K, const int64_t *pos,
                        int64_t R, int64_t d, int64_t n, double scale, int64_t P,
                        double *raw, double *lse, double *work)
{
    for (int64_t j = 0; j < P; ++j)
        raw[j] = 0.0;
    for (int64_t r = 0; r < R; ++r) {
        const int64_t last = pos[r] < n - 1 ? pos[r] : n - 1; /* visible keys [0, last] */
        double mx = -INFINITY;
        for (int64_t j = 0; j <= last; ++j) {
            double dot = 0.0;
            for (int64_t c = 0; c < d; ++c)
                dot += bf16_value(Q[r * d + c]) * bf16_value(K[j * d + c]);
            work[j] = dot * scale;
            if (work[j] > mx)
                mx = work[j];
        }
        double z = 0.0;
        for (int64_t j = 0; j <= last; ++j)
            z += exp(work[j] - mx);
        const double l = mx + log(z);
        if (lse)
            lse[r] = l;
        const int64_t top = last < P - 1 ? last : P - 1;
        for (int64_t j = 0; j <= top; ++j)
            raw[j] += exp(work[j] - l);
    }
}

/* Scores of U independent KV heads.  Q is [U][R][d], K is [U][n][d], raw is
 * [U][P], lse is [U][R] (or NULL).  pos is shared by all units.  Returns 0, or
 * -1 when scratch cannot be allocated. */
int dgeo_scores(const uint16_t *Q, const uint16_t *K, const int64_t *pos, int64_t U,
                int64_t R, int64_t d, int64_t n, double scale, int64_t P, double *raw,
                double *lse)
{
    int failed = 0;
#pragma omp parallel
    {
        double *work = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
        if (!work) {
#pragma omp atomic write
            failed = 1;
        } else {
#pragma omp for schedule(dynamic, 1)
            for (int64_t u = 0; u < U; ++u)
                scores_unit(Q + u * R * d, K + u * n * d, pos, R, d, n, scale, P,
                            raw + u * P, lse ? lse + u * R : NULL, work);
            free(work);
        }
    }
    return failed ? -1 : 0;
}

/*
 * 1D pooling along positions over [0, P) (App. B "maxpool (kernel 7)"):
 * stride 1, half-width r = kernel/2.  MAX takes the max of the in-range cells;
 * AVG sums the in-range cells and divides by the full kernel (zero padding);
 * NONE copies.
 */
int dgeo_pool(const double *raw, int64_t P, int pool, int kernel, double *out)
{
    if (pool != DGEO_POOL_NONE && (kernel < 1 || kernel % 2 == 0))
        return -1;
    const int64_t r = kernel / 2;
    for (int64_t j = 0; j < P; ++j) {
        if (pool == DGEO_POOL_NONE) {
            out[j] = raw[j];
            continue;
        }
        const int64_t lo = j - r < 0 ? 0 : j - r;
        const int64_t hi = j + r > P - 1 ? P - 1 : j + r;
        if (pool == DGEO_POOL_MAX) {
            double mx = -INFINITY;
            for (int64_t i = lo; i <= hi; ++i)
                if (raw[i] > mx)
                    mx = raw[i];
            out[j] = mx;
        } else if (pool == DGEO_POOL_AVG) {
            double s = 0.0;
            for (int64_t i = lo; i <= hi; ++i)
                s += raw[i];
            out[j] = s / (double)kernel;
        } else {
            return -1;
        }
    }
    return 0;
}

typedef struct {
    double score;
    int64_t pos;
} cand_t;

/* Higher score first; equal scores: lower position first. */
static int cand_order(const void *a, const void *b)
{
    const cand_t *x = (const cand_t *)a, *y = (const cand_t *)b;
    if (x->score > y->score)
        return -1;
    if (x->score < y->score)
        return 1;
    return (x->pos > y->pos) - (x->pos < y->pos);
}

static int pos_order(const void *a, const void *b)
{
    const int32_t x = *(const int32_t *)a, y = *(const int32_t *)b;
    return (x > y) - (x < y);
}

/*
 * Retention rule (Alg. 1: I <- R_E(s, B - w), then C[I u window u draft] in
 * temporal order).  Keeps the protected head [0, s0), the `keep` best
 * candidates of [s0, P) by (score desc, position asc), and the protected tail
 * [P, n); writes the s0 + keep + (n - P) positions ascending to idx.
 * scores[j] is indexed by position (only [s0, P) is read).
 * Returns 0, or -1 on bad sizes / allocation failure.
 */
int dgeo_select(const double *scores, int64_t P, int64_t n, int64_t s0, int64_t keep,
                int32_t *idx)
{
    if (s0 < 0 || s0 > P || P > n || keep < 0 || keep > P - s0)
        return -1;
    const int64_t nc = P - s0;
    cand_t *c = (cand_t *)malloc(sizeof(cand_t) * (size_t)(nc > 0 ? nc : 1));
    if (!c)
        return -1;
    for (int64_t j = 0; j < nc; ++j) {
        c[j].score = scores[s0 + j];
        c[j].pos = s0 + j;
    }
    qsort(c, (size_t)nc, sizeof(cand_t), cand_order);
    int64_t o = 0;
    for (int64_t j = 0; j < s0; ++j)
        idx[o++] = (int32_t)j;
    for (int64_t j = 0; j < keep; ++j)
        idx[o + j] = (int32_t)c[j].pos;
    qsort(idx + o, (size_t)keep, sizeof(int32_t), pos_order);
    o += keep;
    for (int64_t j = P; j < n; ++j)
        idx[o++] = (int32_t)j;
    free(c);
    return 0;
}

/*
 * Block-granular retention: the selection ladder's "fixed b-blocks" rung (Table "Selection
 * decomposition"; block sizes 8/16/32 in App. "Diagnostic details").  The paper names the rung
 * but not its rule; this is the reading implemented here.  Candidates [s0, P) form consecutive
 * blocks of bs positions starting at s0 (the last one may be shorter); a block's score is the
 * sum of its positions' scores; blocks are taken whole in the order (score desc, block index
 * asc) while they fit in `keep`, and the first block that does not fit gives its lowest
 * keep - taken positions.  Output as dgeo_select.  bs = 1 is dgeo_select.
 * Returns 0, or -1 on bad sizes / allocation failure.
 */
int dgeo_select_blocks(const double *scores, int64_t P, int64_t n, int64_t s0, int64_t keep,
                       int64_t bs, int32_t *idx)
{
    if (s0 < 0 || s0 > P || P > n || keep < 0 || keep > P - s0 || bs < 1)
        return -1;
    const int64_t nc = P - s0, nb = (nc + bs - 1) / bs;
    cand_t *blk = (cand_t *)malloc(sizeof(cand_t) * (size_t)(nb > 0 ? nb : 1));
    int64_t *take = (int64_t *)calloc((size_t)(nb > 0 ? nb : 1), sizeof(int64_t));
    if (!blk || !take) {
        free(blk);
        free(take);
        return -1;
    }
    for (int64_t k = 0; k < nb; ++k) {
        const int64_t lo = s0 + k * bs, hi = lo + bs < P ? lo + bs : P;
        double sum = 0.0;
        for (int64_t j = lo; j < hi; ++j)
            sum += scores[j];
        blk[k].score = sum;
        blk[k].pos = k;   /* block index: cand_order's tie rule puts the lower block first */
    }
    qsort(blk, (size_t)nb, sizeof(cand_t), cand_order);
    int64_t left = keep;
    for (int64_t i = 0; i < nb && left > 0; ++i) {
        const int64_t k = blk[i].pos, lo = s0 + k * bs;
        const int64_t size = (lo + bs < P ? lo + bs : P) - lo;
        if (size <= left) {
            take[k] = size;
            left -= size;
        } else {
            take[k] = left;
            left = 0;
        }
    }
    int64_t o = 0;
    for (int64_t j = 0; j < s0; ++j)
        idx[o++] = (int32_t)j;
    for (int64_t k = 0; k < nb; ++k)
        for (int64_t q = 0; q < take[k]; ++q)
            idx[o++] = (int32_t)(s0 + k * bs + q);
    for (int64_t j = P; j < n; ++j)
        idx[o++] = (int32_t)j;
    free(blk);
    free(take);
    return 0;
}

/*
 * StreamingLLM retention (App. L): [0, sinks) followed by the last
 * budget - sinks positions.  Returns 0, or -1 on bad sizes.
 */
int dgeo_streaming_indices(int64_t n, int64_t sinks, int64_t budget, int32_t *idx)
{
    if (sinks < 0 || budget < sinks || budget > n)
        return -1;
    int64_t o = 0;
    for (int64_t j = 0; j < sinks; ++j)
        idx[o++] = (int32_t)j;
    for (int64_t j = n - (budget - sinks); j < n; ++j)
        idx[o++] = (int32_t)j;
    return 0;
}

/*
 * Compaction (App. E): out[r] = rows[idx[r]], a byte copy of row_bytes each.
 */
void dgeo_gather(const uint8_t *rows, int64_t row_bytes, const int32_t *idx, int64_t count,
                 uint8_t *out)
{
    for (int64_t r = 0; r < count; ++r)
        memcpy(out + r * row_bytes, rows + (int64_t)idx[r] * row_bytes, (size_t)row_bytes);
}

/*
 * PyramidKV per-layer past budgets (App. L, the discrete schedule):
 * c = B - w, min = floor(c/20), max = 2c - min,
 * steps = floor((max - min)/(L - 1)), out[l] = max - l*steps.
 * Returns 0, or -1 on bad sizes.
 */
int dgeo_pyramid_budgets(int64_t B, int64_t w, int64_t L, int64_t *out)
{
    if (L < 2 || B <= w)
        return -1;
    const int64_t c = B - w;
    const int64_t mn = c / 20;
    const int64_t mx = 2 * c - mn;
    const int64_t steps = (mx - mn) / (L - 1);
    for (int64_t l = 0; l < L; ++l)
        out[l] = mx - l * steps;
    return 0;
}
