/*
 * Fusion staged token adaptation: CPU ORACLE (plain C, double precision).
 *
 * TEST INFRASTRUCTURE ONLY.  The test suite, the smoke check and the CPU-baseline
 * leg of the benchmark are the only callers.  The CUDA library shares no code with
 * this file and never links or calls it.
 *
 * What it computes, one sample at a time, in the paper's order (Sec. III-B: merge
 * first, exit evaluated on merged-but-unpruned tokens, pruning only for samples
 * that continue; Algorithm 1):
 *
 *   merge   Sec. III-C.  Bipartite soft matching after ToMe: the patch tokens are
 *           split into two alternating halves, every token of half A is paired
 *           with its most cosine-similar token of half B, and the r_i best pairs
 *           are averaged into single tokens.  The merge count r_i is a supplied
 *           router output; the average is weighted by token size and the merged
 *           token's size is the sum of its sources' sizes.
 *   exit    Sec. III-D, Eq. 6 and Eq. 7.  p = softmax(head(z)), c = max_k p_k,
 *           exit iff c >= threshold.  The head is LayerNorm(CLS) -> Linear.
 *   prune   Sec. III-E, Eq. 8.  Keep CLS and the top ceil(rho_i * P_i) patch
 *           tokens by score (CLS-attention scores supplied as input).
 *   compact Drop the exited samples (Algorithm 1 returns early for them) and pack
 *           the survivors into a ragged, offset-indexed batch.
 *   exit (MLP heads)  Sec. III-D, Eq. 6 and Eq. 7 with the paper's two exit heads
 *           (Sec. III-G, Sec. IV-I: a SpatialPool head at block 8, a CLS-only head at block 10,
 *           each a 2-layer MLP): head(z) = W2 GELU(W1 LN(pool(z)) + b1) + b2.
 *   attention  the block that consumes a compacted batch (Algorithm 1, Block_b): per
 *           sample and head, softmax(q k^T / sqrt(d_h) + log s_j) v with the size-aware
 *           (proportional) attention of ToMe, so that a merged token of size s weighs
 *           like the s tokens it replaced.
 *   scores  Sec. III-E, Eq. 8 (the prune scores' source): s_i = h_b(z_i) with a
 *           linear scoring head, s = w . z + b for every token, rounded once to
 *           float32.
 *   router  Sec. III-C, Eq. 4 and Eq. 5 (the merge count's source, upstream of
 *           merge): m = sigmoid(w . z_CLS + beta), scaled by the profile ratio
 *           (1 - tau_tgt) / (1 - tau_ref), clamped to [0, 1]; r = floor(m N / 2)
 *           with N the sample's current token count.
 *
 * Readings of points the paper leaves open (fixed here, mirrored by the CUDA path):
 *   - positions within a sample: 0 is CLS, 1..P are patches; half B holds the odd
 *     positions 1,3,5,... (ceil(P/2) tokens), half A the even positions 2,4,...
 *     (floor(P/2) tokens); CLS is in neither half and is never merged;
 *   - cosine similarity uses k / max(||k||_2, 1e-12);
 *   - r_eff = min(max(r_i, 0), |A|); several selected A tokens may share one B
 *     destination, which then averages all of them;
 *   - a merged token's score is the sum of its sources' scores;
 *   - ties: argmax takes the lowest B position, top-r the lowest A position,
 *     top-k pruning the lowest position;
 *   - surviving tokens keep ascending original position, CLS first;
 *   - LayerNorm: biased variance, eps supplied (1e-6 in every workload);
 *   - MLP exit heads: SpatialPool is the size-weighted mean of the patch tokens
 *     (sum s_t x_t / sum s_t; the CLS row when a sample has no patch), GELU is the
 *     erf form, and for bf16 the LayerNorm output and the hidden activations are
 *     rounded to bf16 (the operands of the two products);
 *   - bf16 storage: keys enter the dot products as stored; the LayerNorm output
 *     is rounded to bf16 before the head; merged tokens are rounded to bf16 once,
 *     after the weighted mean; everything else is accumulated in double.
 *
 * Each function also reports decision margins (best minus runner-up), so that a
 * parity test can count the decisions that lie closer than its threshold.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_F32 0
#define ORC_BF16 1

#define ORC_OK 0
#define ORC_ERR_ARG -1
#define ORC_ERR_NOMEM -2

/* ------------------------------------------------------------------------- */
/* storage conversions                                                        */
/* ------------------------------------------------------------------------- */

/* bf16 bit pattern -> exact double. */
static double bf16_to_double(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Round a double to the nearest bfloat16 value, ties to even, in one step
 * (bfloat16 keeps 8 significant bits and float32's exponent range). */
static uint16_t double_to_bf16(double v)
{
    if (isnan(v))
        return 0x7FC0;
    uint16_t sign = signbit(v) ? 0x8000 : 0;
    double a = fabs(v);
    if (a == 0.0)
        return sign;
    if (isinf(a))
        return (uint16_t)(sign | 0x7F80);
    int e;
    frexp(a, &e);                /* 2^(e-1) <= a < 2^e */
    int lead = e - 1;
    if (lead < -126)
        lead = -126;             /* subnormal range: fixed spacing 2^-133 */
    double spacing = ldexp(1.0, lead - 7);
    double q = a / spacing;      /* exact: scaling by a power of two */
    double whole = floor(q);
    double frac = q - whole;
    if (frac > 0.5 || (frac == 0.5 && fmod(whole, 2.0) == 1.0))
        whole += 1.0;
    double rv = whole * spacing;
    if (rv > 0x1.FEp127)         /* beyond the largest finite bfloat16 */
        return (uint16_t)(sign | 0x7F80);
    float f = (float)rv;         /* exact: at most 8 significant bits */
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return (uint16_t)(sign | ((u >> 16) & 0x7FFF));
}

static double load_elem(int dtype, const void *base, int64_t idx)
{
    if (dtype == ORC_BF16)
        return bf16_to_double(((const uint16_t *)base)[idx]);
    return (double)((const float *)base)[idx];
}

static void store_elem(int dtype, void *base, int64_t idx, double v)
{
    if (dtype == ORC_BF16)
        ((uint16_t *)base)[idx] = double_to_bf16(v);
    else
        ((float *)base)[idx] = (float)v;
}

/* Expose the two conversions so that the tests can pin them. */
uint16_t orc_double_to_bf16(double v) { return double_to_bf16(v); }
double orc_bf16_to_double(uint16_t h) { return bf16_to_double(h); }

/* Sort idx[0..n) so that val[idx[.]] is decreasing, equal values by increasing
 * index (insertion sort: slow, stable and obviously correct). */
static void order_desc(const double *val, int *idx, int n)
{
    for (int i = 0; i < n; ++i)
        idx[i] = i;
    for (int i = 1; i < n; ++i) {
        int cur = idx[i];
        int j = i - 1;
        while (j >= 0 && (val[idx[j]] < val[cur] || (val[idx[j]] == val[cur] && idx[j] > cur))) {
            idx[j + 1] = idx[j];
            --j;
        }
        idx[j + 1] = cur;
    }
}

/* ------------------------------------------------------------------------- */
/* merge (Sec. III-C)                                                          */
/* ------------------------------------------------------------------------- */

/*
 * x, keys: [T, d] and [T, dk] (bf16 bits or f32); sizes, scores: [T] f32 (scores may be
 * NULL); r: [B] merge counts.  Outputs, all host memory owned by the caller:
 *   x_out [T', d], sizes_out [T'], scores_out [T'] (NULL when scores is NULL),
 *   offsets_out [B+1], keep_idx [T'] (input row of each output row),
 *   dst_map [T] (output row each input row went to or was merged into),
 *   a_match [T] (for A tokens: input row of the matched B token; -1 otherwise),
 *   argmax_gap [T] (A tokens: best minus runner-up cosine; +inf otherwise),
 *   topr_gap [B] (r-th minus (r+1)-th best-match similarity; +inf if no boundary).
 */
int orc_merge(int dtype, int B, const int32_t *offsets, int d, const void *x,
              const void *keys, int dk, const float *sizes, const float *scores,
              const int32_t *r, void *x_out, float *sizes_out, float *scores_out,
              int32_t *offsets_out, int32_t *keep_idx, int32_t *dst_map, int32_t *a_match,
              double *argmax_gap, double *topr_gap)
{
    if (B < 0 || d <= 0 || dk <= 0)
        return ORC_ERR_ARG;
    offsets_out[0] = 0;
    for (int i = 0; i < B; ++i) {
        const int64_t base = offsets[i];
        const int N = offsets[i + 1] - offsets[i];
        if (N < 1)
            return ORC_ERR_ARG;
        const int P = N - 1;
        const int nA = P / 2;
        const int nB = (P + 1) / 2;

        double *khat = malloc(sizeof(double) * (size_t)N * (size_t)dk);
        double *best = malloc(sizeof(double) * (size_t)(nA + 1));
        int *match = malloc(sizeof(int) * (size_t)(nA + 1));
        int *order = malloc(sizeof(int) * (size_t)(nA + 1));
        int *selected = calloc((size_t)(nA + 1), sizeof(int));
        int *out_local = malloc(sizeof(int) * (size_t)N);
        double *num = malloc(sizeof(double) * (size_t)d);
        if (!khat || !best || !match || !order || !selected || !out_local || !num)
            return ORC_ERR_NOMEM;

        /* L2-normalised keys */
        for (int p = 0; p < N; ++p) {
            double ss = 0.0;
            for (int j = 0; j < dk; ++j) {
                double v = load_elem(dtype, keys, (base + p) * dk + j);
                ss += v * v;
            }
            double nrm = sqrt(ss);
            double inv = 1.0 / (nrm > 1e-12 ? nrm : 1e-12);
            for (int j = 0; j < dk; ++j)
                khat[(int64_t)p * dk + j] = load_elem(dtype, keys, (base + p) * dk + j) * inv;
        }

        /* each A token (position 2+2m) -> most cosine-similar B token (position 1+2n) */
        for (int m = 0; m < nA; ++m) {
            const int pa = 2 + 2 * m;
            double bv = -INFINITY, second = -INFINITY;
            int bn = -1;
            for (int n = 0; n < nB; ++n) {
                const int pb = 1 + 2 * n;
                double s = 0.0;
                for (int j = 0; j < dk; ++j)
                    s += khat[(int64_t)pa * dk + j] * khat[(int64_t)pb * dk + j];
                if (s > bv) {
                    second = bv;
                    bv = s;
                    bn = n;
                } else if (s > second) {
                    second = s;
                }
            }
            best[m] = bv;
            match[m] = bn;
            if (argmax_gap)
                argmax_gap[base + pa] = (nB >= 2) ? bv - second : INFINITY;
        }

        /* the r_eff best pairs are merged */
        int r_eff = r[i];
        if (r_eff < 0)
            r_eff = 0;
        if (r_eff > nA)
            r_eff = nA;
        order_desc(best, order, nA);
        for (int q = 0; q < r_eff; ++q)
            selected[order[q]] = 1;
        if (topr_gap)
            topr_gap[i] = (r_eff > 0 && r_eff < nA) ? best[order[r_eff - 1]] - best[order[r_eff]]
                                                    : INFINITY;

        /* survivors keep ascending position: CLS, B tokens and unselected A tokens */
        int n_out = 0;
        for (int p = 0; p < N; ++p) {
            int is_a = (p >= 2 && p % 2 == 0);
            out_local[p] = (is_a && selected[(p - 2) / 2]) ? -1 : n_out++;
        }
        const int64_t obase = offsets_out[i];
        offsets_out[i + 1] = (int32_t)(obase + n_out);

        for (int p = 0; p < N; ++p) {
            int is_a = (p >= 2 && p % 2 == 0);
            int dst = out_local[p];
            if (is_a && selected[(p - 2) / 2])
                dst = out_local[1 + 2 * match[(p - 2) / 2]];
            if (dst_map)
                dst_map[base + p] = (int32_t)(obase + dst);
            if (a_match)
                a_match[base + p] = is_a ? (int32_t)(base + 1 + 2 * match[(p - 2) / 2]) : -1;
        }

        /* size-weighted scatter-mean into each destination */
        for (int p = 0; p < N; ++p) {
            const int o = out_local[p];
            if (o < 0)
                continue;
            double wsum = sizes[base + p];
            double ssum = scores ? scores[base + p] : 0.0;
            for (int j = 0; j < d; ++j)
                num[j] = (double)sizes[base + p] * load_elem(dtype, x, (base + p) * d + j);
            if (p % 2 == 1) {                       /* a B token may receive A tokens */
                const int n = (p - 1) / 2;
                for (int m = 0; m < nA; ++m) {
                    if (!selected[m] || match[m] != n)
                        continue;
                    const int64_t ra = base + 2 + 2 * m;
                    wsum += sizes[ra];
                    if (scores)
                        ssum += scores[ra];
                    for (int j = 0; j < d; ++j)
                        num[j] += (double)sizes[ra] * load_elem(dtype, x, ra * d + j);
                }
            }
            const int64_t orow = obase + o;
            /* a token with no merged sources comes out unchanged: size*x/size == x exactly */
            for (int j = 0; j < d; ++j)
                store_elem(dtype, x_out, orow * d + j, num[j] / wsum);
            sizes_out[orow] = (float)wsum;
            if (scores && scores_out)
                scores_out[orow] = (float)ssum;
            if (keep_idx)
                keep_idx[orow] = (int32_t)(base + p);
        }

        free(khat);
        free(best);
        free(match);
        free(order);
        free(selected);
        free(out_local);
        free(num);
    }
    return ORC_OK;
}

/* ------------------------------------------------------------------------- */
/* exit check (Sec. III-D, Eq. 6-7)                                           */
/* ------------------------------------------------------------------------- */

/*
 * Reads the CLS row (first row) of every sample.  gamma, beta: [d]; W: [C, d] row-major
 * (all in dtype); bias: [C] f32.  Outputs: exit_mask [B], logits [B, C] f32 (every row),
 * max_prob [B], exit_gap [B] = |c - tau|, u_out [B, d] (the head input after the bf16
 * rounding, as double; may be NULL).
 */
int orc_exit(int dtype, int B, const int32_t *offsets, int d, const void *x,
             const void *gamma, const void *beta, double eps, const void *W,
             const float *bias, int C, double tau, uint8_t *exit_mask, float *logits,
             float *max_prob, double *exit_gap, double *u_out)
{
    if (B < 0 || d <= 0 || C <= 0)
        return ORC_ERR_ARG;
    double *u = malloc(sizeof(double) * (size_t)d);
    double *l = malloc(sizeof(double) * (size_t)C);
    if (!u || !l)
        return ORC_ERR_NOMEM;
    for (int i = 0; i < B; ++i) {
        const int64_t row = offsets[i];
        double mean = 0.0;
        for (int j = 0; j < d; ++j)
            mean += load_elem(dtype, x, row * d + j);
        mean /= d;
        double var = 0.0;
        for (int j = 0; j < d; ++j) {
            double t = load_elem(dtype, x, row * d + j) - mean;
            var += t * t;
        }
        var /= d;
        const double rstd = 1.0 / sqrt(var + eps);
        for (int j = 0; j < d; ++j) {
            double v = (load_elem(dtype, x, row * d + j) - mean) * rstd * load_elem(dtype, gamma, j) +
                       load_elem(dtype, beta, j);
            if (dtype == ORC_BF16)
                v = bf16_to_double(double_to_bf16(v));
            u[j] = v;
            if (u_out)
                u_out[(int64_t)i * d + j] = v;
        }
        double lmax = -INFINITY;
        for (int k = 0; k < C; ++k) {
            double acc = 0.0;
            for (int j = 0; j < d; ++j)
                acc += load_elem(dtype, W, (int64_t)k * d + j) * u[j];
            l[k] = acc + (double)bias[k];
            if (l[k] > lmax)
                lmax = l[k];
        }
        double S = 0.0;
        for (int k = 0; k < C; ++k)
            S += exp(l[k] - lmax);
        const double c = 1.0 / S;   /* max_k softmax(l)_k */
        if (exit_mask)
            exit_mask[i] = (c >= tau) ? 1 : 0;
        if (max_prob)
            max_prob[i] = (float)c;
        if (exit_gap)
            exit_gap[i] = fabs(c - tau);
        if (logits)
            for (int k = 0; k < C; ++k)
                logits[(int64_t)i * C + k] = (float)l[k];
    }
    free(u);
    free(l);
    return ORC_OK;
}

/* ------------------------------------------------------------------------- */
/* prune (Sec. III-E, Eq. 8)                                                  */
/* ------------------------------------------------------------------------- */

/*
 * Keeps CLS plus the k_i = ceil(rho_i * P_i) highest-scored patches of every sample
 * (k clamped to [0, P_i]), in ascending position.  Outputs as in orc_merge;
 * prune_gap [B] = k-th minus (k+1)-th score (+inf if no boundary).
 */
int orc_prune(int dtype, int B, const int32_t *offsets, int d, const void *x,
              const float *sizes, const float *scores, const float *rho, void *x_out,
              float *sizes_out, float *scores_out, int32_t *offsets_out, int32_t *keep_idx,
              double *prune_gap)
{
    if (B < 0 || d <= 0)
        return ORC_ERR_ARG;
    offsets_out[0] = 0;
    for (int i = 0; i < B; ++i) {
        const int64_t base = offsets[i];
        const int N = offsets[i + 1] - offsets[i];
        if (N < 1)
            return ORC_ERR_ARG;
        const int P = N - 1;
        double kk = ceil((double)rho[i] * (double)P);
        int k = kk < 0.0 ? 0 : (kk > P ? P : (int)kk);

        double *s = malloc(sizeof(double) * (size_t)(P + 1));
        int *order = malloc(sizeof(int) * (size_t)(P + 1));
        int *kept = calloc((size_t)(P + 1), sizeof(int));
        if (!s || !order || !kept)
            return ORC_ERR_NOMEM;
        for (int q = 0; q < P; ++q)
            s[q] = (double)scores[base + 1 + q];
        order_desc(s, order, P);
        for (int q = 0; q < k; ++q)
            kept[order[q]] = 1;
        if (prune_gap)
            prune_gap[i] = (k > 0 && k < P) ? s[order[k - 1]] - s[order[k]] : INFINITY;

        int64_t orow = offsets_out[i];
        for (int p = 0; p < N; ++p) {
            if (p > 0 && !kept[p - 1])
                continue;
            for (int j = 0; j < d; ++j)
                store_elem(dtype, x_out, orow * d + j, load_elem(dtype, x, (base + p) * d + j));
            sizes_out[orow] = sizes[base + p];
            if (scores_out)
                scores_out[orow] = scores[base + p];
            if (keep_idx)
                keep_idx[orow] = (int32_t)(base + p);
            ++orow;
        }
        offsets_out[i + 1] = (int32_t)orow;
        free(s);
        free(order);
        free(kept);
    }
    return ORC_OK;
}

/* ------------------------------------------------------------------------- */
/* compact (Algorithm 1: exited samples leave the batch)                      */
/* ------------------------------------------------------------------------- */

/*
 * Survivors (exit_mask == 0) keep ascending sample order.  ids: [B] original sample ids
 * (NULL = 0..B-1).  Outputs: x_out, sizes_out, scores_out (NULL when scores is NULL),
 * offsets_out [B'+1], ids_out [B'], keep_idx [T'], *n_out = B'.
 */
int orc_compact(int dtype, int B, const int32_t *offsets, int d, const void *x,
                const float *sizes, const float *scores, const uint8_t *exit_mask,
                const int32_t *ids, void *x_out, float *sizes_out, float *scores_out,
                int32_t *offsets_out, int32_t *ids_out, int32_t *keep_idx, int32_t *n_out)
{
    if (B < 0 || d <= 0)
        return ORC_ERR_ARG;
    int j = 0;
    offsets_out[0] = 0;
    for (int i = 0; i < B; ++i) {
        if (exit_mask[i])
            continue;
        const int64_t base = offsets[i];
        const int N = offsets[i + 1] - offsets[i];
        int64_t orow = offsets_out[j];
        for (int p = 0; p < N; ++p, ++orow) {
            for (int q = 0; q < d; ++q)
                store_elem(dtype, x_out, orow * d + q, load_elem(dtype, x, (base + p) * d + q));
            sizes_out[orow] = sizes[base + p];
            if (scores && scores_out)
                scores_out[orow] = scores[base + p];
            if (keep_idx)
                keep_idx[orow] = (int32_t)(base + p);
        }
        offsets_out[j + 1] = (int32_t)orow;
        ids_out[j] = ids ? ids[i] : i;
        ++j;
    }
    *n_out = j;
    return ORC_OK;
}

/* ------------------------------------------------------------------------- */
/* merge router with profile scaling (Sec. III-C, Eq. 4 and Eq. 5)             */
/* ------------------------------------------------------------------------- */
/*
 * For every sample i (rows offsets[i]..offsets[i+1]-1, CLS first):
 *   m_i  = sigmoid(w . z_i + beta)                          (Eq. 4, z_i the CLS row)
 *   mt_i = m_i * (1 - tau_tgt) / (1 - tau_ref), clamped to [0, 1]   (Eq. 5)
 *   r_i  = floor(mt_i * N_i / 2), N_i the sample's token count, CLS included
 * Outputs are indexed by the sample's original id (ids[i], or i when ids is NULL):
 * r_out, mt_out (may be NULL) and r_gap (may be NULL) = distance of mt_i N_i / 2 to
 * the nearest integer, the margin of the floor decision.  tau_ref must be below 1.
 */
int orc_merge_router(int dtype, int B, const int32_t *offsets, const int32_t *ids, int d, const void *x,
                     const void *w, double beta, double tau_tgt, double tau_ref, int32_t *r_out,
                     double *mt_out, double *r_gap)
{
    if (B < 0 || d <= 0 || !(tau_ref < 1.0))
        return ORC_ERR_ARG;
    const double scale = (1.0 - tau_tgt) / (1.0 - tau_ref);
    for (int i = 0; i < B; ++i) {
        const int64_t row = offsets[i];
        const int N = offsets[i + 1] - offsets[i];
        double z = 0.0;
        for (int j = 0; j < d; ++j)
            z += load_elem(dtype, w, j) * load_elem(dtype, x, row * d + j);
        const double m = 1.0 / (1.0 + exp(-(z + beta)));
        double mt = m * scale;
        if (mt < 0.0)
            mt = 0.0;
        if (mt > 1.0)
            mt = 1.0;
        const double v = mt * (0.5 * (double)N);
        const double r = floor(v);
        const int id = ids ? ids[i] : i;
        r_out[id] = (int32_t)r;
        if (mt_out)
            mt_out[id] = mt;
        if (r_gap) {
            const double f = v - r;
            r_gap[id] = f < 1.0 - f ? f : 1.0 - f;
        }
    }
    return ORC_OK;
}

/* ------------------------------------------------------------------------- */
/* pruning router: token scores (Sec. III-E, Eq. 8)                             */
/* ------------------------------------------------------------------------- */
/*
 * s_t = w . z_t + b for every token row t of the B samples (rows offsets[0] ..
 * offsets[B] - 1), accumulated in double and rounded once to float32.  Rows outside
 * the samples are not written.
 */
int orc_token_scores(int dtype, int B, const int32_t *offsets, int d, const void *x, const void *w, double b,
                     float *scores_out)
{
    if (B < 0 || d <= 0)
        return ORC_ERR_ARG;
    for (int i = 0; i < B; ++i)
        for (int64_t t = offsets[i]; t < offsets[i + 1]; ++t) {
            double acc = 0.0;
            for (int j = 0; j < d; ++j)
                acc += load_elem(dtype, w, j) * load_elem(dtype, x, t * d + j);
            scores_out[t] = (float)(acc + b);
        }
    return ORC_OK;
}

/* ------------------------------------------------------------------------- */
/* exit check with the MLP heads (Sec. III-D, Eq. 6-7; Sec. III-G, Sec. IV-I)     */
/* ------------------------------------------------------------------------- */
/*
 * head(z) = W2 GELU(W1 LN(pool(z)) + b1) + b2, c = max_k softmax(head(z))_k, exit iff
 * c >= tau.  pool 0 (CLS-only head): the CLS row; pool 1 (SpatialPool head): the
 * size-weighted mean of the patch rows (positions 1..N-1), the CLS row when N = 1.
 * GELU(a) = a (1 + erf(a / sqrt 2)) / 2.  W1 [H, d] and W2 [C, H] row-major, gamma and
 * beta [d], all in dtype; b1 [H], b2 [C] f32.  Outputs as in orc_exit, plus pool_out
 * [B, d] and hidden_out [B, H] (after the bf16 rounding; both double, may be NULL).
 */
int orc_exit_mlp(int dtype, int B, const int32_t *offsets, int d, const void *x, const float *sizes, int pool,
                 const void *gamma, const void *beta, double eps, const void *W1, const float *b1, int H,
                 const void *W2, const float *b2, int C, double tau, uint8_t *exit_mask, float *logits,
                 float *max_prob, double *exit_gap, double *pool_out, double *hidden_out)
{
    if (B < 0 || d <= 0 || H <= 0 || C <= 0 || (pool != 0 && pool != 1))
        return ORC_ERR_ARG;
    double *z = malloc(sizeof(double) * (size_t)d);
    double *u = malloc(sizeof(double) * (size_t)d);
    double *h = malloc(sizeof(double) * (size_t)H);
    double *l = malloc(sizeof(double) * (size_t)C);
    if (!z || !u || !h || !l) {
        free(z);
        free(u);
        free(h);
        free(l);
        return ORC_ERR_NOMEM;
    }
    for (int i = 0; i < B; ++i) {
        const int64_t o = offsets[i], n = offsets[i + 1] - offsets[i];
        /* pool */
        if (pool == 0 || n < 2) {
            for (int j = 0; j < d; ++j)
                z[j] = load_elem(dtype, x, o * d + j);
        } else {
            double wsum = 0.0;
            for (int j = 0; j < d; ++j)
                z[j] = 0.0;
            for (int64_t t = o + 1; t < o + n; ++t) {
                wsum += (double)sizes[t];
                for (int j = 0; j < d; ++j)
                    z[j] += (double)sizes[t] * load_elem(dtype, x, t * d + j);
            }
            for (int j = 0; j < d; ++j)
                z[j] /= wsum;
        }
        if (pool_out)
            memcpy(pool_out + (int64_t)i * d, z, sizeof(double) * (size_t)d);
        /* LayerNorm */
        double mean = 0.0;
        for (int j = 0; j < d; ++j)
            mean += z[j];
        mean /= d;
        double var = 0.0;
        for (int j = 0; j < d; ++j)
            var += (z[j] - mean) * (z[j] - mean);
        var /= d;
        const double rstd = 1.0 / sqrt(var + eps);
        for (int j = 0; j < d; ++j) {
            double v = (z[j] - mean) * rstd * load_elem(dtype, gamma, j) + load_elem(dtype, beta, j);
            if (dtype == ORC_BF16)
                v = bf16_to_double(double_to_bf16(v));
            u[j] = v;
        }
        /* first layer and GELU */
        for (int k = 0; k < H; ++k) {
            double a = 0.0;
            for (int j = 0; j < d; ++j)
                a += load_elem(dtype, W1, (int64_t)k * d + j) * u[j];
            a += (double)b1[k];
            double g = 0.5 * a * (1.0 + erf(a / sqrt(2.0)));
            if (dtype == ORC_BF16)
                g = bf16_to_double(double_to_bf16(g));
            h[k] = g;
            if (hidden_out)
                hidden_out[(int64_t)i * H + k] = g;
        }
        /* second layer, softmax maximum, exit rule */
        double lmax = -INFINITY;
        for (int c = 0; c < C; ++c) {
            double acc = 0.0;
            for (int k = 0; k < H; ++k)
                acc += load_elem(dtype, W2, (int64_t)c * H + k) * h[k];
            l[c] = acc + (double)b2[c];
            if (l[c] > lmax)
                lmax = l[c];
        }
        double S = 0.0;
        for (int c = 0; c < C; ++c)
            S += exp(l[c] - lmax);
        const double cmax = 1.0 / S;
        if (exit_mask)
            exit_mask[i] = (cmax >= tau) ? 1 : 0;
        if (max_prob)
            max_prob[i] = (float)cmax;
        if (exit_gap)
            exit_gap[i] = fabs(cmax - tau);
        if (logits)
            for (int c = 0; c < C; ++c)
                logits[(int64_t)i * C + c] = (float)l[c];
    }
    free(z);
    free(u);
    free(h);
    free(l);
    return ORC_OK;
}

/* ------------------------------------------------------------------------- */
/* size-aware attention over a ragged batch (Algorithm 1, Block_b; ToMe)         */
/* ------------------------------------------------------------------------- */
/*
 * qkv [rows, 3, H, dh] row-major (the q, k and v projections of every token, dtype);
 * sizes [rows] float32, or NULL for plain attention (every size 1).  For every sample,
 * head h and query row m of the sample:
 *   l_j = (q_m . k_j) / sqrt(dh) + log(s_j),  p = softmax(l) over the sample's rows,
 *   out[m, h, :] = sum_j p_j v_j   (double, [rows, H, dh]; rows outside the samples untouched).
 */
int orc_attention(int dtype, int B, const int32_t *offsets, int H, int dh, const void *qkv, const float *sizes,
                  double *out)
{
    if (B < 0 || H <= 0 || dh <= 0)
        return ORC_ERR_ARG;
    const int64_t rs = (int64_t)3 * H * dh; /* row stride of qkv */
    const double scale = 1.0 / sqrt((double)dh);
    for (int i = 0; i < B; ++i) {
        const int64_t o = offsets[i], n = offsets[i + 1] - offsets[i];
        double *l = malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
        if (!l)
            return ORC_ERR_NOMEM;
        for (int h = 0; h < H; ++h) {
            const int64_t qo = (int64_t)h * dh, ko = (int64_t)(H + h) * dh, vo = (int64_t)(2 * H + h) * dh;
            for (int64_t m = 0; m < n; ++m) {
                double lmax = -INFINITY;
                for (int64_t j = 0; j < n; ++j) {
                    double dot = 0.0;
                    for (int e = 0; e < dh; ++e)
                        dot += load_elem(dtype, qkv, (o + m) * rs + qo + e) * load_elem(dtype, qkv, (o + j) * rs + ko + e);
                    l[j] = dot * scale + (sizes ? log((double)sizes[o + j]) : 0.0);
                    if (l[j] > lmax)
                        lmax = l[j];
                }
                double S = 0.0;
                for (int64_t j = 0; j < n; ++j) {
                    l[j] = exp(l[j] - lmax);
                    S += l[j];
                }
                double *dst = out + (o + m) * (int64_t)H * dh + (int64_t)h * dh;
                for (int e = 0; e < dh; ++e) {
                    double acc = 0.0;
                    for (int64_t j = 0; j < n; ++j)
                        acc += l[j] * load_elem(dtype, qkv, (o + j) * rs + vo + e);
                    dst[e] = acc / S;
                }
            }
        }
        free(l);
    }
    return ORC_OK;
}
