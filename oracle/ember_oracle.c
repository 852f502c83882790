/*
 * ember_oracle.c -- plain, slow CPU restatement of the Ember optimizer step.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the parity oracle for the CUDA
 * library in paper_2607_01455_gb300/csrc.  It shares no source, header,
 * helper or constant with that library and is never linked into it.  Only the
 * test suite, the smoke check of __graft_entry__ and the CPU-baseline leg of
 * bench.py load it.  The product path must never call it.
 *
 * What it computes: Algorithm 1 ("Ember") of "Token Geometry"
 * (arXiv 2607.01455, Section 2.1), taken in the algorithm's own order:
 *
 *   r_t = beta2 r_{t-1} + (1-beta2) mean_j(g_t^2)      row second moment
 *   c_t = beta2 c_{t-1} + (1-beta2) mean_i(g_t^2)      column second moment
 *   rhat = r_t / (1 - beta2^t),  chat = c_t / (1 - beta2^t)   bias correction
 *   s_t  = sqrt( mean(rhat) * mean(chat) )               geometric-mean normaliser
 *   vtil = rhat chat^T / s_t                              factored preconditioner
 *   theta_t = theta_{t-1} -/+ alpha g_t / (sqrt(vtil) + eps)   update
 *
 * Precision and readings of the paper:
 *   - all arithmetic is fp64; sums run in plain index order;
 *   - the state vectors r (V floats) and c (D floats) are stored as fp32,
 *     which is how the paper's model-scaling table of Section 3.1 counts
 *     them; the rest of the step uses the stored fp32 values;
 *   - the weights are rounded once per step to their storage type (fp32 or
 *     bfloat16) with round-to-nearest-even;
 *   - the paper ascends a reward; this oracle descends a loss by default
 *     (maximize=0 gives theta - alpha u, maximize=1 gives theta + alpha u).
 *     The denominator depends on g only through g^2, so the two coincide
 *     under g -> -g;
 *   - when s_t == 0 (every statistic is zero) the preconditioner is taken as
 *     zero, so u = g / eps, which is 0 because g is then zero;
 *   - the sparse step (Section 2.2) is the dense step on the gradient obtained
 *     by summing, per token id, the rows of every occurrence of that id, in
 *     occurrence order.  Ids outside [0, V) contribute nothing.
 *   - variant ROW uses vtil_ij = rhat_i and variant COL uses vtil_ij = chat_j
 *     (the ablation rows of the Section 2.1 table); bias_correction = 0 uses
 *     rhat = r, chat = c (the bias-correction ablation of the appendix).
 *
 * Built with gcc -O2 -fno-fast-math -ffp-contract=off so that every
 * operation rounds exactly as written.  The timed CPU baseline also builds
 * it with -fopenmp: the row loops and the blocks of the column loop then run
 * on all host cores, and since every sum keeps its order (each row's sum
 * over its columns, each column's sum over the rows in index order) that
 * build gives the same bits.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_FULL 0
#define ORC_ROW 1
#define ORC_COL 2

#define ORC_COL_BLOCK 64 /* columns per block of the column-sum loop */

#define ORC_OK 0
#define ORC_EINVAL -1
#define ORC_ENOMEM -2

/* ------------------------------------------------------------------ */
/* bfloat16 storage: 1 sign bit, 8 exponent bits (binary32's range),   */
/* 8 significant bits.  Conversions written from that definition.      */
/* ------------------------------------------------------------------ */

static double bf16_bits_to_double(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16; /* a bfloat16 is the top half of a binary32 */
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Round a double to the nearest bfloat16, ties to even. */
static uint16_t double_to_bf16_bits(double x)
{
    if (isnan(x))
        return (uint16_t)0x7FC0u;
    uint16_t sign = signbit(x) ? (uint16_t)0x8000u : (uint16_t)0u;
    double a = fabs(x);
    if (a == 0.0)
        return sign;
    if (isinf(a))
        return (uint16_t)(sign | 0x7F80u);
    int e;
    frexp(a, &e);                 /* a = m 2^e with m in [0.5, 1) */
    int lead = e - 1;             /* floor(log2 a) */
    if (lead < -126)
        lead = -126;              /* subnormal range: fixed quantum */
    double quantum = ldexp(1.0, lead - 7); /* spacing of 8-bit significands */
    double q = rint(a / quantum); /* exact scaling; rint rounds ties to even */
    double y = q * quantum;
    if (y >= 0x1p128)             /* past the largest finite bfloat16 */
        return (uint16_t)(sign | 0x7F80u);
    float f = (float)y;           /* exact: y has at most 8 significant bits */
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return (uint16_t)(sign | (uint16_t)((u >> 16) & 0x7FFFu));
}

void ember_oracle_round_bf16(int64_t n, const double *x, uint16_t *out)
{
    for (int64_t k = 0; k < n; ++k)
        out[k] = double_to_bf16_bits(x[k]);
}

void ember_oracle_bf16_to_double(int64_t n, const uint16_t *x, double *out)
{
    for (int64_t k = 0; k < n; ++k)
        out[k] = bf16_bits_to_double(x[k]);
}

/* ------------------------------------------------------------------ */
/* One Ember step on a dense V x D gradient (Algorithm 1).             */
/* The gradient is read either from fp32 (Gf) or fp64 (Gd) storage.    */
/* ------------------------------------------------------------------ */

static double grad_at(const float *Gf, const double *Gd, int64_t k)
{
    return Gf ? (double)Gf[k] : Gd[k];
}

static double weight_at(const void *W, int w_is_bf16, int64_t k)
{
    if (w_is_bf16)
        return bf16_bits_to_double(((const uint16_t *)W)[k]);
    return (double)((const float *)W)[k];
}

static void weight_store(void *W, int w_is_bf16, int64_t k, double x)
{
    if (w_is_bf16)
        ((uint16_t *)W)[k] = double_to_bf16_bits(x);
    else
        ((float *)W)[k] = (float)x; /* C conversion rounds to nearest even */
}

/* diag (optional, 5 doubles): bias-correction denominator 1-beta2^t,
 * mean(rhat), mean(chat), s, and the number of rows whose r is zero. */
static int alg1_step(int64_t V, int64_t D, int w_is_bf16, void *W,
                     const float *Gf, const double *Gd, float *r, float *c,
                     double lr, int64_t t, double beta2, double eps,
                     int maximize, int bias_correction, int variant,
                     double *diag)
{
    if (V < 1 || D < 1 || t < 1 || !(beta2 >= 0.0 && beta2 < 1.0) ||
        !(eps >= 0.0) || variant < ORC_FULL || variant > ORC_COL)
        return ORC_EINVAL;

    /* Row second moment: r_i <- beta2 r_i + (1-beta2) mean_j g_ij^2. */
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < V; ++i) {
        double sum = 0.0;
        for (int64_t j = 0; j < D; ++j) {
            double g = grad_at(Gf, Gd, i * D + j);
            sum += g * g;
        }
        double mean_row = sum / (double)D;
        r[i] = (float)(beta2 * (double)r[i] + (1.0 - beta2) * mean_row);
    }

    /* Column second moment: c_j <- beta2 c_j + (1-beta2) mean_i g_ij^2. */
    double *colsum = (double *)calloc((size_t)D, sizeof(double));
    if (!colsum)
        return ORC_ENOMEM;
    /* Each column's sum runs over the rows in index order; the columns are
       independent, so they are taken in blocks (in parallel under OpenMP). */
    #pragma omp parallel for schedule(static)
    for (int64_t jb = 0; jb < D; jb += ORC_COL_BLOCK) {
        int64_t je = (jb + ORC_COL_BLOCK < D) ? jb + ORC_COL_BLOCK : D;
        for (int64_t i = 0; i < V; ++i)
            for (int64_t j = jb; j < je; ++j) {
                double g = grad_at(Gf, Gd, i * D + j);
                colsum[j] += g * g;
            }
    }
    for (int64_t j = 0; j < D; ++j) {
        double mean_col = colsum[j] / (double)V;
        c[j] = (float)(beta2 * (double)c[j] + (1.0 - beta2) * mean_col);
    }
    free(colsum);

    /* Bias correction: rhat = r / (1 - beta2^t), chat = c / (1 - beta2^t). */
    double bc = bias_correction ? 1.0 - pow(beta2, (double)t) : 1.0;

    /* Geometric-mean normaliser: s = sqrt(mean(rhat) * mean(chat)). */
    double rbar = 0.0, cbar = 0.0;
    int64_t zero_rows = 0;
    for (int64_t i = 0; i < V; ++i) {
        rbar += (double)r[i] / bc;
        zero_rows += (r[i] == 0.0f);
    }
    rbar /= (double)V;
    for (int64_t j = 0; j < D; ++j)
        cbar += (double)c[j] / bc;
    cbar /= (double)D;
    double s = sqrt(rbar * cbar);

    /* Preconditioner vtil = rhat chat^T / s, never stored; update. */
    #pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < V; ++i) {
        double rhat = (double)r[i] / bc;
        for (int64_t j = 0; j < D; ++j) {
            double chat = (double)c[j] / bc;
            double vtil;
            if (variant == ORC_ROW)
                vtil = rhat;
            else if (variant == ORC_COL)
                vtil = chat;
            else
                vtil = (s > 0.0) ? rhat * chat / s : 0.0;
            int64_t k = i * D + j;
            double g = grad_at(Gf, Gd, k);
            double u = g / (sqrt(vtil) + eps);
            double w = weight_at(W, w_is_bf16, k);
            weight_store(W, w_is_bf16, k, maximize ? w + lr * u : w - lr * u);
        }
    }

    if (diag) {
        diag[0] = bc;
        diag[1] = rbar;
        diag[2] = cbar;
        diag[3] = s;
        diag[4] = (double)zero_rows;
    }
    return ORC_OK;
}

int ember_oracle_step_dense(int64_t V, int64_t D, int w_is_bf16, void *W,
                            const float *G, float *r, float *c, double lr,
                            int64_t t, double beta2, double eps, int maximize,
                            int bias_correction, int variant, double *diag)
{
    if (!W || !G || !r || !c)
        return ORC_EINVAL;
    return alg1_step(V, D, w_is_bf16, W, G, NULL, r, c, lr, t, beta2, eps,
                     maximize, bias_correction, variant, diag);
}

/* Threads of the OpenMP build: n > 0 sets the count; returns the count in
 * use (always 1 in the plain build). */
int ember_oracle_threads(int n)
{
#ifdef _OPENMP
    if (n > 0)
        omp_set_num_threads(n);
    return omp_get_max_threads();
#else
    (void)n;
    return 1;
#endif
}

/* ------------------------------------------------------------------ */
/* Sparse step (Section 2.2): an embedding gradient has nonzero rows    */
/* only for the token ids of the batch; an id seen k times receives the */
/* sum of its k per-occurrence rows.  The step is then Algorithm 1 on   */
/* that V x D gradient.                                                */
/* ------------------------------------------------------------------ */

int ember_oracle_step_sparse(int64_t V, int64_t D, int w_is_bf16, void *W,
                             int64_t N, const int64_t *ids, const float *rows,
                             float *r, float *c, double lr, int64_t t,
                             double beta2, double eps, int maximize,
                             int bias_correction, int variant, double *diag)
{
    if (!W || !r || !c || V < 1 || D < 1 || N < 0 || (N > 0 && (!ids || !rows)))
        return ORC_EINVAL;
    double *Gd = (double *)calloc((size_t)V * (size_t)D, sizeof(double));
    if (!Gd)
        return ORC_ENOMEM;
    for (int64_t k = 0; k < N; ++k) {
        int64_t id = ids[k];
        if (id < 0 || id >= V)
            continue;
        for (int64_t j = 0; j < D; ++j)
            Gd[id * D + j] += (double)rows[k * D + j];
    }
    int rc = alg1_step(V, D, w_is_bf16, W, NULL, Gd, r, c, lr, t, beta2, eps,
                       maximize, bias_correction, variant, diag);
    free(Gd);
    return rc;
}

/* Token-id dedup: the distinct valid ids in ascending order and how often
 * each occurs.  Returns U, or a negative code. */
static int cmp_i64(const void *a, const void *b)
{
    int64_t x = *(const int64_t *)a, y = *(const int64_t *)b;
    return (x > y) - (x < y);
}

int64_t ember_oracle_dedup(int64_t N, const int64_t *ids, int64_t V,
                           int64_t *uniq, int64_t *counts)
{
    if (N < 0 || V < 1 || (N > 0 && (!ids || !uniq || !counts)))
        return ORC_EINVAL;
    int64_t *tmp = (int64_t *)malloc((size_t)(N > 0 ? N : 1) * sizeof(int64_t));
    if (!tmp)
        return ORC_ENOMEM;
    int64_t n = 0;
    for (int64_t k = 0; k < N; ++k)
        if (ids[k] >= 0 && ids[k] < V)
            tmp[n++] = ids[k];
    qsort(tmp, (size_t)n, sizeof(int64_t), cmp_i64);
    int64_t U = 0;
    for (int64_t k = 0; k < n; ++k) {
        if (U > 0 && uniq[U - 1] == tmp[k]) {
            counts[U - 1] += 1;
        } else {
            uniq[U] = tmp[k];
            counts[U] = 1;
            ++U;
        }
    }
    free(tmp);
    return U;
}

/* ------------------------------------------------------------------ */
/* LM-head gradient, the step that produces G for an output head       */
/* (appendix "Decomposing the Squared Gradient"): token t contributes  */
/* the outer product of its output-side error delta_t (V values, the   */
/* softmax error) and its hidden state h_t (D values); the batch        */
/* gradient is the sum over the T tokens, G = dlogits^T H, i.e.        */
/*   G[v][d] = sum_t dlogits[t][v] * hidden[t][d].                     */
/* Inputs are bfloat16 bit patterns, row-major T x V and T x D.  Each  */
/* product and the sum over t (in token order) are taken in fp64.      */
/* rows: the nrows row indices v to compute (NULL: all V rows, in      */
/* order); G and absG receive nrows x D values.  absG (optional) gets   */
/* sum_t |dlogits[t][v] hidden[t][d]|, the scale against which the    */
/* rounding of any other summation order is bounded.                   */
/* ------------------------------------------------------------------ */

int ember_oracle_lmhead_grad(int64_t T, int64_t V, int64_t D,
                             const uint16_t *dlogits, const uint16_t *hidden,
                             int64_t nrows, const int64_t *rows,
                             double *G, double *absG)
{
    if (T < 0 || V < 1 || D < 1 || !G || (T > 0 && (!dlogits || !hidden)))
        return ORC_EINVAL;
    if (!rows)
        nrows = V;
    if (nrows < 0)
        return ORC_EINVAL;
    double *hrow = (double *)malloc((size_t)D * sizeof(double));
    if (!hrow)
        return ORC_ENOMEM;
    for (int64_t q = 0; q < nrows; ++q) {
        int64_t v = rows ? rows[q] : q;
        if (v < 0 || v >= V) {
            free(hrow);
            return ORC_EINVAL;
        }
        double *out = G + q * D;
        double *aout = absG ? absG + q * D : NULL;
        for (int64_t d = 0; d < D; ++d) {
            out[d] = 0.0;
            if (aout)
                aout[d] = 0.0;
        }
        for (int64_t t = 0; t < T; ++t) {
            double delta = bf16_bits_to_double(dlogits[t * V + v]);
            for (int64_t d = 0; d < D; ++d)
                hrow[d] = bf16_bits_to_double(hidden[t * D + d]);
            for (int64_t d = 0; d < D; ++d) {
                double p = delta * hrow[d];
                out[d] += p;
                if (aout)
                    aout[d] += fabs(p);
            }
        }
    }
    free(hrow);
    return ORC_OK;
}
