/*
 * sc_oracle.c -- plain fp64 CPU oracle for SparseCoder's sparse attention with
 * learned token pruning (arXiv 2310.07109).
 *
 * THIS IS TEST INFRASTRUCTURE.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load it.  It shares no code, header, table
 * or helper with the CUDA library; the product path never calls it.
 *
 * What it computes, per sequence and layer, over the n tokens that survived
 * the previous layer (current index c = 0..n-1, original position p(c)):
 *
 *   1. Allowed key set of query row i (Sec. "Sparse Attention": token i is
 *      attended by units i-w .. i+w; Sec. "Extractor of Attention Scores":
 *      special tokens attend to every other token, and every token attends to
 *      them):
 *          A(i) = {0..n-1}                               if i is global
 *          A(i) = {j : |i - j| <= w}  U  {global j}      otherwise
 *      A token is global when its ORIGINAL position is in the global set G.
 *   2. S_h[i,j] = q_{i,h} . k_{j,h} / sqrt(d) for j in A(i)   (Sec. "Attention
 *      Mechanisms of Transformers": scaled dot-product self-attention).
 *   3. Row-wise softmax over A(i) (Fig. 1 caption: softmax is taken per row),
 *      O_h[i] = sum_j P_h[i,j] v_{j,h}.
 *   4. Importance score: the attention probabilities are accumulated
 *      vertically (Sec. "Pruning"; Fig. 1 caption), averaged over heads and
 *      query rows:   s_j = (1 / (H n)) * sum_h sum_i P_h[i,j].
 *   5. Binarised keep mask (Sec. "Token Pruning", Step 2): token j is kept when
 *      s_j >= theta; the first current token (the CLS token) is always kept.
 *      Kept tokens are removed/compacted in order (Step 3, hard pruning).
 *      Two alternatives to the per-layer threshold alpha_l / n_l, both from the
 *      paper: an absolute threshold theta_l per layer (Sec. "RQ4": the
 *      thresholds of the layers are scaled linearly up to the last one), and
 *      the "top-k of the sequence length" family of Sec. "Pruning": a layer
 *      keeps k = ceil(rho_l n) tokens (clamped to 1..n), the first token and
 *      the k-1 others with the largest scores, ties going to the lower index.
 *
 * Everything is double precision and loops over the definition directly; no
 * blocking, no online softmax, no reordering.  The stack driver reads the
 * bf16 bit patterns of Q/K/V and widens them exactly to double.
 *
 * Readings of the paper that this file fixes (the paper is silent or
 * inconsistent on them): the window is +-w inclusive (2w+1 keys); the window
 * is measured in the current (compacted) index; the keep test is ">=";
 * theta_l = alpha_l / n_l per sequence; only the first current token is
 * force-kept, other global tokens obey the threshold and stay global while
 * they survive.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define SCO_EXPORT __attribute__((visibility("default")))

/* ------------------------------------------------------------------------ */
/* allowed-set predicate, step 1                                             */
/* ------------------------------------------------------------------------ */
static int allowed(int w, const int *is_global, int i, int j)
{
    if (is_global[i]) return 1;
    if (is_global[j]) return 1;
    int dist = i > j ? i - j : j - i;
    return dist <= w;
}

/* ------------------------------------------------------------------------ */
/* one head of one layer: steps 2-4 for every row                            */
/* ------------------------------------------------------------------------ */
typedef struct {
    int n, H, d, w;
    const double *Q, *K, *V;   /* [n][H][d] */
    const int *is_global;      /* [n] */
    double *O;                 /* [n][H][d] or NULL */
    double *colsum;            /* [H][n]: sum_i P_h[i,j] for this head */
    int h_begin, h_end;
} head_job;

static double dot(const double *a, const double *b, int d)
{
    double s = 0.0;
    for (int t = 0; t < d; ++t) s += a[t] * b[t];
    return s;
}

static void *run_heads(void *arg)
{
    head_job *jb = (head_job *)arg;
    const int n = jb->n, H = jb->H, d = jb->d;
    const double scale = 1.0 / sqrt((double)d);
    double *srow = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    for (int h = jb->h_begin; h < jb->h_end; ++h) {
        double *cs = jb->colsum + (size_t)h * n;
        for (int j = 0; j < n; ++j) cs[j] = 0.0;
        for (int i = 0; i < n; ++i) {
            const double *qi = jb->Q + ((size_t)i * H + h) * d;
            /* scores over the allowed set, max for a stable exp */
            double mx = -INFINITY;
            for (int j = 0; j < n; ++j) {
                if (!allowed(jb->w, jb->is_global, i, j)) continue;
                const double *kj = jb->K + ((size_t)j * H + h) * d;
                srow[j] = dot(qi, kj, d) * scale;
                if (srow[j] > mx) mx = srow[j];
            }
            double z = 0.0;
            for (int j = 0; j < n; ++j) {
                if (!allowed(jb->w, jb->is_global, i, j)) continue;
                srow[j] = exp(srow[j] - mx);
                z += srow[j];
            }
            double *oi = jb->O ? jb->O + ((size_t)i * H + h) * d : NULL;
            if (oi) for (int t = 0; t < d; ++t) oi[t] = 0.0;
            for (int j = 0; j < n; ++j) {
                if (!allowed(jb->w, jb->is_global, i, j)) continue;
                double p = srow[j] / z;
                cs[j] += p;
                if (oi) {
                    const double *vj = jb->V + ((size_t)j * H + h) * d;
                    for (int t = 0; t < d; ++t) oi[t] += p * vj[t];
                }
            }
        }
    }
    free(srow);
    return NULL;
}

/* Runs the heads of one layer on up to nthreads threads and returns the
 * per-head column sums in colsum[H][n]. */
static int layer_heads(int n, int H, int d, int w, const double *Q,
                       const double *K, const double *V, const int *is_global,
                       double *O, double *colsum, int nthreads)
{
    if (nthreads < 1) nthreads = 1;
    if (nthreads > H) nthreads = H;
    head_job jobs[64];
    pthread_t tids[64];
    if (nthreads > 64) nthreads = 64;
    int per = (H + nthreads - 1) / nthreads;
    int used = 0;
    for (int t = 0; t < nthreads; ++t) {
        int hb = t * per, he = hb + per;
        if (he > H) he = H;
        if (hb >= he) break;
        head_job jb = {n, H, d, w, Q, K, V, is_global, O, colsum, hb, he};
        jobs[used] = jb;
        ++used;
    }
    for (int t = 1; t < used; ++t)
        if (pthread_create(&tids[t], NULL, run_heads, &jobs[t]) != 0)
            run_heads(&jobs[t]), tids[t] = 0;
    if (used > 0) run_heads(&jobs[0]);
    for (int t = 1; t < used; ++t)
        if (tids[t]) pthread_join(tids[t], NULL);
    return used;
}

/* ------------------------------------------------------------------------ */
/* one layer: steps 1-5                                                      */
/* ------------------------------------------------------------------------ */
/*
 * Q, K, V   [n][H][d] current order.
 * is_global [n] 1 when the token's original position is a global position.
 * theta     absolute keep threshold.
 * O         [n][H][d] output (may be NULL).
 * scores    [n] output s_j.
 * keep      [n] output 0/1.
 * Returns the number of kept tokens, or -1 on bad arguments.
 */
SCO_EXPORT int sco_layer(int n, int H, int d, int w, const double *Q,
                         const double *K, const double *V,
                         const int *is_global, double theta, double *O,
                         double *scores, int *keep, int nthreads)
{
    if (n < 0 || H < 1 || d < 1 || w < 0) return -1;
    if (n == 0) return 0;
    double *colsum = (double *)malloc(sizeof(double) * (size_t)H * n);
    if (!colsum) return -1;
    layer_heads(n, H, d, w, Q, K, V, is_global, O, colsum, nthreads);
    int kept = 0;
    for (int j = 0; j < n; ++j) {
        double acc = 0.0;
        for (int h = 0; h < H; ++h) acc += colsum[(size_t)h * n + j];
        scores[j] = acc / ((double)H * (double)n);
        keep[j] = (j == 0) || (scores[j] >= theta);
        kept += keep[j];
    }
    free(colsum);
    return kept;
}

/* ------------------------------------------------------------------------ */
/* top-ratio keep rule (Sec. "Pruning", second family)                      */
/* ------------------------------------------------------------------------ */
/* k = ceil(rho * n), clamped to 1..n.  rho * n is exact in double for a rho
 * that came from a float and n < 2^24. */
SCO_EXPORT int sco_top_count(double rho, int n)
{
    if (n <= 0) return 0;
    double c = ceil(rho * (double)n);
    if (!(c >= 1.0)) return 1;   /* also a NaN ratio */
    if (c >= (double)n) return n;
    return (int)c;
}

/*
 * keep[j] for the top-ratio rule: token 0, and each other token whose rank
 * among tokens 1..n-1 (larger score first, ties by lower index) is below k-1.
 * The rank is counted directly: the number of other tokens that come first.
 * Returns the number kept (k), or -1 on bad arguments.
 */
SCO_EXPORT int sco_keep_top(int n, const double *scores, int k, int *keep)
{
    if (n < 0 || k < 0) return -1;
    if (n == 0) return 0;
    if (k < 1) k = 1;
    if (k > n) k = n;
    keep[0] = 1;
    for (int j = 1; j < n; ++j) {
        int rank = 0;
        for (int i = 1; i < n; ++i)
            if (scores[i] > scores[j] || (scores[i] == scores[j] && i < j)) ++rank;
        keep[j] = rank < k - 1;
    }
    return k;
}

/*
 * Sampled evaluation of one layer, for sizes where the full layer is too slow:
 * O rows of the listed query rows, and s_j of the listed key columns, each
 * computed directly from the definition (a column sums P_h[i,j] over every
 * row i whose allowed set contains j, each row with its own full softmax).
 */
static double row_prob(int n, int H, int d, int w, const double *Q,
                       const double *K, const int *is_global, int h, int i,
                       int jsel, double *srow)
{
    const double scale = 1.0 / sqrt((double)d);
    const double *qi = Q + ((size_t)i * H + h) * d;
    double mx = -INFINITY;
    for (int j = 0; j < n; ++j) {
        if (!allowed(w, is_global, i, j)) continue;
        srow[j] = dot(qi, K + ((size_t)j * H + h) * d, d) * scale;
        if (srow[j] > mx) mx = srow[j];
    }
    double z = 0.0;
    for (int j = 0; j < n; ++j) {
        if (!allowed(w, is_global, i, j)) continue;
        z += exp(srow[j] - mx);
    }
    return exp(srow[jsel] - mx) / z;
}

SCO_EXPORT int sco_layer_sampled(int n, int H, int d, int w, const double *Q,
                                 const double *K, const double *V,
                                 const int *is_global, const int *rows,
                                 int nrows, double *O_rows, const int *cols,
                                 int ncols, double *s_cols)
{
    if (n < 1 || H < 1 || d < 1 || w < 0) return -1;
    double *srow = (double *)malloc(sizeof(double) * (size_t)n);
    const double scale = 1.0 / sqrt((double)d);
    for (int r = 0; r < nrows; ++r) {
        int i = rows[r];
        if (i < 0 || i >= n) { free(srow); return -1; }
        for (int h = 0; h < H; ++h) {
            const double *qi = Q + ((size_t)i * H + h) * d;
            double mx = -INFINITY;
            for (int j = 0; j < n; ++j) {
                if (!allowed(w, is_global, i, j)) continue;
                srow[j] = dot(qi, K + ((size_t)j * H + h) * d, d) * scale;
                if (srow[j] > mx) mx = srow[j];
            }
            double z = 0.0;
            for (int j = 0; j < n; ++j) {
                if (!allowed(w, is_global, i, j)) continue;
                srow[j] = exp(srow[j] - mx);
                z += srow[j];
            }
            double *o = O_rows + ((size_t)r * H + h) * d;
            for (int t = 0; t < d; ++t) o[t] = 0.0;
            for (int j = 0; j < n; ++j) {
                if (!allowed(w, is_global, i, j)) continue;
                const double *vj = V + ((size_t)j * H + h) * d;
                for (int t = 0; t < d; ++t) o[t] += (srow[j] / z) * vj[t];
            }
        }
    }
    for (int c = 0; c < ncols; ++c) {
        int j = cols[c];
        if (j < 0 || j >= n) { free(srow); return -1; }
        double acc = 0.0;
        for (int h = 0; h < H; ++h)
            for (int i = 0; i < n; ++i)
                if (allowed(w, is_global, i, j))
                    acc += row_prob(n, H, d, w, Q, K, is_global, h, i, j, srow);
        s_cols[c] = acc / ((double)H * (double)n);
    }
    free(srow);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* the layer stack                                                           */
/* ------------------------------------------------------------------------ */
static double bf16_to_double(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static int is_global_position(const int *g, int ng, int p)
{
    for (int t = 0; t < ng; ++t)
        if (g[t] == p) return 1;
    return 0;
}

/*
 * n_layers layers over B sequences of padded length L.
 * Qb, Kb, Vb  bf16 bit patterns [n_layers][B][L][H][d], indexed by ORIGINAL
 *             position: layer l reads the rows of the tokens that survived
 *             layers 0..l-1.
 * pad_mask    [B][L] (1 = real token) or NULL.  Padding tokens are removed
 *             before the first layer (Fig. "experiment" caption: inputs are
 *             padded to max_length; padding carries no content).
 * gpos, ngpos global original positions.
 * alpha       [n_layers]: the keep rule's value per layer.
 * rule        0: theta_l = alpha_l / n_l for each sequence;
 *             1: theta_l = alpha_l (absolute);
 *             2: top ratio rho_l = alpha_l (see sco_keep_top).
 * O           [n_layers][B][L][H][d] doubles at current slots, or NULL.
 * scores      [n_layers][B][L] doubles at current slots.
 * pos         [n_layers+1][B][L] original positions of the current tokens.
 * len         [n_layers+1][B] current lengths.
 * Slots at or beyond the current length are left untouched.
 */
SCO_EXPORT int sco_stack(int n_layers, int B, int L, int H, int d, int w,
                         const uint16_t *Qb, const uint16_t *Kb,
                         const uint16_t *Vb, const uint8_t *pad_mask,
                         const int *gpos, int ngpos, const double *alpha,
                         int rule, double *O, double *scores, int *pos,
                         int *len, int nthreads)
{
    if (n_layers < 1 || B < 1 || L < 1 || H < 1 || d < 1 || w < 0) return -1;
    if (rule < 0 || rule > 2) return -1;
    const size_t row = (size_t)H * d;
    double *q = (double *)malloc(sizeof(double) * (size_t)L * row);
    double *k = (double *)malloc(sizeof(double) * (size_t)L * row);
    double *v = (double *)malloc(sizeof(double) * (size_t)L * row);
    double *o = (double *)malloc(sizeof(double) * (size_t)L * row);
    double *s = (double *)malloc(sizeof(double) * (size_t)L);
    int *keep = (int *)malloc(sizeof(int) * (size_t)L);
    int *isg = (int *)malloc(sizeof(int) * (size_t)L);
    if (!q || !k || !v || !o || !s || !keep || !isg) return -1;

    for (int b = 0; b < B; ++b) {
        /* padding pre-prune */
        int *pos0 = pos + (size_t)b * L;
        int n = 0;
        for (int p = 0; p < L; ++p)
            if (!pad_mask || pad_mask[(size_t)b * L + p]) pos0[n++] = p;
        len[b] = n;
        for (int l = 0; l < n_layers; ++l) {
            const int *pl = pos + ((size_t)l * B + b) * L;
            int *pn = pos + ((size_t)(l + 1) * B + b) * L;
            size_t base = (size_t)l * B + b;
            /* gather the current tokens' rows (original-position order) */
            for (int c = 0; c < n; ++c) {
                size_t src = (base * L + (size_t)pl[c]) * row;
                for (size_t t = 0; t < row; ++t) {
                    q[(size_t)c * row + t] = bf16_to_double(Qb[src + t]);
                    k[(size_t)c * row + t] = bf16_to_double(Kb[src + t]);
                    v[(size_t)c * row + t] = bf16_to_double(Vb[src + t]);
                }
                isg[c] = is_global_position(gpos, ngpos, pl[c]);
            }
            double theta = rule == 1 ? alpha[l] : (n > 0 ? alpha[l] / (double)n : 0.0);
            sco_layer(n, H, d, w, q, k, v, isg, theta, o, s, keep, nthreads);
            if (rule == 2) sco_keep_top(n, s, sco_top_count(alpha[l], n), keep);
            int m = 0;
            for (int c = 0; c < n; ++c) {
                scores[base * L + c] = s[c];
                if (O)
                    memcpy(O + (base * L + c) * row, o + (size_t)c * row,
                           sizeof(double) * row);
                if (keep[c]) pn[m++] = pl[c];
            }
            n = m;
            len[(size_t)(l + 1) * B + b] = n;
        }
    }
    free(q); free(k); free(v); free(o); free(s); free(keep); free(isg);
    return 0;
}
