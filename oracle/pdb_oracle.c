/*
 * pdb_oracle.c -- plain, slow, single-threaded CPU oracle for
 * serially-equivalent sparse SGD (data-centric synchronization).
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the bench's
 * CPU-baseline leg may load this file.  It shares no code, header, table or
 * constant generator with the CUDA library; both sides implement the same
 * written numerics independently.
 *
 * What it computes, and where the paper defines it:
 *   - the parameter database M(Theta, D): D (CSR rows) immutable, Theta (w)
 *     mutable                                               -- Definition 1
 *   - chunks = single features, read/write set of example t = its nonzero
 *     features                                        -- Definitions 2 and 3
 *   - the sequential computation: iterations run one after another, each
 *     reads all of its chunks before writing any       -- Algorithm 1, Def. 4
 *     one iteration = one training example (Section 6.3: "1 training sample
 *     versus the entire dataset"); the update is the scalar gradient step of
 *     Section 2 applied to that example's loss term f_t.
 *   - per-chunk iteration numbers of the read protocol (Section 5) become
 *     per-feature occurrence chains: prev/next occurrence and occurrence rank
 *   - dependency levels: a level is one barrier-separated step of
 *     non-conflicting transactions (Theorem 3), level = longest conflict path
 *   - the BSP comparison: reads of a batch see the snapshot taken at the read
 *     barrier, writes apply after the write barrier (Algorithm 2a)
 *
 * Floating point follows one written rule set (no contraction: compile with
 * -ffp-contract=off and no fast-math):
 *   dot(t):  32 partial sums a[0..31] = +0; element i of the row (CSR order)
 *            does a[i mod 32] = fmaf(w[col], val, a[i mod 32]); then for
 *            off = 16, 8, 4, 2, 1 every a[l] becomes a[l] + a[l xor off];
 *            the margin is a[0].
 *   grad:    logistic  g = -y / (1 + expf_cw(y*m))
 *            squared   g = m - y                  (loss (m - y)^2 / 2)
 *            hinge     g = (y*m < 1) ? -y : 0     (subgradient 0 at y*m = 1)
 *   update:  c = eta*g;  w_j = w_j - c*x_j        (each op one fp32 rounding)
 *   expf_cw: Cody-Waite reduction x = k ln2 + r (Cody and Waite, "Software
 *            Manual for the Elementary Functions", 1980) with k = rint(x*log2e),
 *            ln2 split into a 16-bit head and a tail; e^r by its degree-7
 *            Taylor polynomial (coefficients 1/n!) in fmaf Horner form; 2^k
 *            applied as two exact power-of-two factors.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_OK 0
#define ORC_BAD_ROWPTR 1
#define ORC_BAD_COL 2
#define ORC_DUP 3
#define ORC_NOMEM 4

#define ORC_LOGISTIC 0
#define ORC_SQUARED 1
#define ORC_HINGE 2

/* ------------------------------------------------------------------ checks */

/* Definition 1: D is a set of examples; Definition 3: the read set of an
 * iteration is a set of chunks, so a feature may appear once per row. */
int orc_validate(int64_t n_rows, int64_t n_cols, int64_t nnz, const int64_t *row_ptr, const int32_t *col)
{
    if (n_rows < 0 || n_cols < 0 || nnz < 0) return ORC_BAD_ROWPTR;
    if (row_ptr[0] != 0 || row_ptr[n_rows] != nnz) return ORC_BAD_ROWPTR;
    for (int64_t t = 0; t < n_rows; ++t)
        if (row_ptr[t + 1] < row_ptr[t]) return ORC_BAD_ROWPTR;
    for (int64_t p = 0; p < nnz; ++p)
        if (col[p] < 0 || (int64_t)col[p] >= n_cols) return ORC_BAD_COL;
    int64_t *seen = (int64_t *)malloc(sizeof(int64_t) * (size_t)(n_cols > 0 ? n_cols : 1));
    if (!seen) return ORC_NOMEM;
    for (int64_t j = 0; j < n_cols; ++j) seen[j] = -1;
    int rc = ORC_OK;
    for (int64_t t = 0; t < n_rows && rc == ORC_OK; ++t)
        for (int64_t p = row_ptr[t]; p < row_ptr[t + 1]; ++p) {
            if (seen[col[p]] == t) { rc = ORC_DUP; break; }
            seen[col[p]] = t;
        }
    free(seen);
    return rc;
}

/* ------------------------------------------------------------------ chains */

/* Per-feature occurrence chains, the sparse form of the read protocol's
 * per-chunk iteration number (Section 5): walking the examples in data order,
 * each occurrence p of feature j links to the previous occurrence of j
 * (prev), the previous one links forward to p (next), and rank[p] counts the
 * occurrences of j before p.  csc_pos lists, feature by feature, the
 * positions of its occurrences in data order; feat_ptr delimits the features. */
int orc_chains(int64_t n_rows, int64_t n_cols, int64_t nnz, const int64_t *row_ptr, const int32_t *col,
               int32_t *csc_pos, int64_t *feat_ptr, int32_t *prev, int32_t *next, int32_t *rank)
{
    (void)n_rows;
    (void)row_ptr;
    int64_t *last = (int64_t *)malloc(sizeof(int64_t) * (size_t)(n_cols > 0 ? n_cols : 1));
    int64_t *cnt = (int64_t *)calloc((size_t)(n_cols > 0 ? n_cols : 1), sizeof(int64_t));
    if (!last || !cnt) { free(last); free(cnt); return ORC_NOMEM; }
    for (int64_t j = 0; j < n_cols; ++j) last[j] = -1;
    for (int64_t p = 0; p < nnz; ++p) {
        int32_t j = col[p];
        prev[p] = (int32_t)last[j];
        next[p] = -1;
        if (last[j] >= 0) next[last[j]] = (int32_t)p;
        rank[p] = (int32_t)cnt[j];
        cnt[j] += 1;
        last[j] = p;
    }
    feat_ptr[0] = 0;
    for (int64_t j = 0; j < n_cols; ++j) feat_ptr[j + 1] = feat_ptr[j] + cnt[j];
    for (int64_t p = 0; p < nnz; ++p) csc_pos[feat_ptr[col[p]] + rank[p]] = (int32_t)p;
    free(last);
    free(cnt);
    return ORC_OK;
}

/* ------------------------------------------------------------------ levels */

/* Dependency level of every example (Theorem 3: one level is one BSP step
 * over transactions with pairwise disjoint chunk sets).  level[t] is the
 * length of the longest chain of conflicting earlier examples ending at t:
 * level[t] = 1 + max over occurrences p of row t with a previous occurrence
 * of level[row of prev[p]], and 0 when no feature of t occurred before.
 * Returns the number of levels L = 1 + max level (0 for no rows). */
int64_t orc_levels(int64_t n_rows, int64_t nnz, const int64_t *row_ptr, const int32_t *prev, int32_t *level)
{
    int32_t *row_of = (int32_t *)malloc(sizeof(int32_t) * (size_t)(nnz > 0 ? nnz : 1));
    if (!row_of) return -1;
    for (int64_t t = 0; t < n_rows; ++t)
        for (int64_t p = row_ptr[t]; p < row_ptr[t + 1]; ++p) row_of[p] = (int32_t)t;
    int64_t n_levels = 0;
    for (int64_t t = 0; t < n_rows; ++t) {
        int32_t lv = -1;
        for (int64_t p = row_ptr[t]; p < row_ptr[t + 1]; ++p)
            if (prev[p] >= 0 && level[row_of[prev[p]]] > lv) lv = level[row_of[prev[p]]];
        level[t] = lv + 1;
        if (level[t] + 1 > n_levels) n_levels = level[t] + 1;
    }
    free(row_of);
    return n_levels;
}

/* Examples grouped by level, ascending example id inside a level (a stable
 * counting sort); level_ptr[l] .. level_ptr[l+1] delimits level l. */
int orc_level_order(int64_t n_rows, int64_t n_levels, const int32_t *level, int32_t *order, int64_t *level_ptr)
{
    for (int64_t l = 0; l <= n_levels; ++l) level_ptr[l] = 0;
    for (int64_t t = 0; t < n_rows; ++t) level_ptr[level[t] + 1] += 1;
    for (int64_t l = 0; l < n_levels; ++l) level_ptr[l + 1] += level_ptr[l];
    int64_t *fill = (int64_t *)malloc(sizeof(int64_t) * (size_t)(n_levels > 0 ? n_levels : 1));
    if (!fill) return ORC_NOMEM;
    for (int64_t l = 0; l < n_levels; ++l) fill[l] = level_ptr[l];
    for (int64_t t = 0; t < n_rows; ++t) order[fill[level[t]]++] = (int32_t)t;
    free(fill);
    return ORC_OK;
}

/* ------------------------------------------------------------------ numerics */

/* expf_cw of the rule set above: the exponential of the logistic gradient.
 * The paper fixes none; this one is written from Cody and Waite's range
 * reduction and the Taylor series, so both sides can compute it alike. */
float orc_expf(float x)
{
    const float log2e = (float)1.4426950408889634074;
    const float ln2_hi = 0.693145751953125f;              /* 45426 / 2^16 */
    const float ln2_lo = (float)(0.6931471805599453094 - 0.693145751953125);
    if (x != x) return x;
    if (x > 89.0f) x = 89.0f;
    if (x < -104.0f) x = -104.0f;
    float kf = rintf(x * log2e);
    float r = x - kf * ln2_hi;
    r = r - kf * ln2_lo;
    float p = (float)(1.0 / 5040.0);
    p = fmaf(p, r, (float)(1.0 / 720.0));
    p = fmaf(p, r, (float)(1.0 / 120.0));
    p = fmaf(p, r, (float)(1.0 / 24.0));
    p = fmaf(p, r, (float)(1.0 / 6.0));
    p = fmaf(p, r, 0.5f);
    p = fmaf(p, r, 1.0f);
    p = fmaf(p, r, 1.0f);
    int k = (int)kf;
    int h = k / 2;
    int k2 = k - h;
    union { uint32_t u; float f; } s1, s2;
    s1.u = (uint32_t)(h + 127) << 23;
    s2.u = (uint32_t)(k2 + 127) << 23;
    return (p * s1.f) * s2.f;
}

void orc_expf_n(const float *x, float *out, int64_t n)
{
    for (int64_t i = 0; i < n; ++i) out[i] = orc_expf(x[i]);
}

/* margin m_t = w . x_t in the fixed 32-partial-sum order */
float orc_dot(const float *w, const int32_t *col, const float *val, int64_t k)
{
    float a[32], b[32];
    for (int l = 0; l < 32; ++l) a[l] = 0.0f;
    for (int64_t i = 0; i < k; ++i) a[i % 32] = fmaf(w[col[i]], val ? val[i] : 1.0f, a[i % 32]);
    for (int off = 16; off >= 1; off >>= 1) {
        for (int l = 0; l < 32; ++l) b[l] = a[l] + a[l ^ off];
        for (int l = 0; l < 32; ++l) a[l] = b[l];
    }
    return a[0];
}

/* derivative of the example's loss term f_t with respect to its margin (the
 * scalar of the gradient step of Section 2, per example) */
float orc_grad(int loss, float m, float y)
{
    if (loss == ORC_LOGISTIC) return -y / (1.0f + orc_expf(y * m));
    if (loss == ORC_SQUARED) return m - y;
    return (y * m < 1.0f) ? -y : 0.0f;
}

/* ------------------------------------------------------------------ SGD */

/* One SGD transaction on example t (Definition 3: all reads of its chunks,
 * the fixed-point computation, then all writes). */
static void sgd_step(int64_t t, const int64_t *row_ptr, const int32_t *col, const float *val, const float *y,
                     float *w, int loss, float eta)
{
    int64_t b = row_ptr[t], k = row_ptr[t + 1] - row_ptr[t];
    float m = orc_dot(w, col + b, val ? val + b : NULL, k);
    float c = eta * orc_grad(loss, m, y[t]);
    for (int64_t i = 0; i < k; ++i) {
        float x = val ? val[b + i] : 1.0f;
        w[col[b + i]] = w[col[b + i]] - c * x;
    }
}

/* Algorithm 1 with one iteration per example, for n_epochs passes over D.
 * order == NULL runs the examples in data order; otherwise order[0..N) is the
 * order of execution (Theorem 2: any order that keeps every conflicting pair
 * in data order gives the same model). */
int orc_sgd(int64_t n_rows, const int64_t *row_ptr, const int32_t *col, const float *val, const float *y,
            float *w, int loss, float eta, int n_epochs, const int32_t *order)
{
    for (int e = 0; e < n_epochs; ++e)
        for (int64_t i = 0; i < n_rows; ++i) sgd_step(order ? order[i] : i, row_ptr, col, val, y, w, loss, eta);
    return ORC_OK;
}

/* Algorithm 2a with a batch of B examples between the barriers: every
 * example of the batch reads the snapshot w_b (read barrier), then every
 * feature j takes delta_j = sum over the batch's examples, ascending, of
 * c_i * x_ij and w_j = w_j - delta_j (write barrier).  The last batch may be
 * short.  B = 1 is the per-example BSP of Theorem 1. */
int orc_bsp(int64_t n_rows, int64_t n_cols, const int64_t *row_ptr, const int32_t *col, const float *val,
            const float *y, float *w, int loss, float eta, int64_t batch, int n_epochs)
{
    if (batch < 1) return ORC_BAD_ROWPTR;
    float *c = (float *)malloc(sizeof(float) * (size_t)batch);
    float *delta = (float *)calloc((size_t)(n_cols > 0 ? n_cols : 1), sizeof(float));
    if (!c || !delta) { free(c); free(delta); return ORC_NOMEM; }
    for (int e = 0; e < n_epochs; ++e)
        for (int64_t b0 = 0; b0 < n_rows; b0 += batch) {
            int64_t b1 = b0 + batch < n_rows ? b0 + batch : n_rows;
            for (int64_t t = b0; t < b1; ++t) {
                int64_t b = row_ptr[t], k = row_ptr[t + 1] - b;
                float m = orc_dot(w, col + b, val ? val + b : NULL, k);
                c[t - b0] = eta * orc_grad(loss, m, y[t]);
            }
            for (int64_t t = b0; t < b1; ++t)
                for (int64_t p = row_ptr[t]; p < row_ptr[t + 1]; ++p)
                    delta[col[p]] = delta[col[p]] + c[t - b0] * (val ? val[p] : 1.0f);
            for (int64_t t = b0; t < b1; ++t)
                for (int64_t p = row_ptr[t]; p < row_ptr[t + 1]; ++p) {
                    w[col[p]] = w[col[p]] - delta[col[p]];
                    delta[col[p]] = 0.0f;
                }
        }
    free(c);
    free(delta);
    return ORC_OK;
}

/* The same sequential SGD in fp64 with libm exp and a plain left-to-right
 * dot product: a drift reference for the fp32 result, not a parity target. */
int orc_sgd_f64(int64_t n_rows, const int64_t *row_ptr, const int32_t *col, const float *val, const float *y,
                double *w, int loss, double eta, int n_epochs)
{
    for (int e = 0; e < n_epochs; ++e)
        for (int64_t t = 0; t < n_rows; ++t) {
            double m = 0.0;
            for (int64_t p = row_ptr[t]; p < row_ptr[t + 1]; ++p) m += w[col[p]] * (val ? (double)val[p] : 1.0);
            double yy = y[t], g;
            if (loss == ORC_LOGISTIC) g = -yy / (1.0 + exp(yy * m));
            else if (loss == ORC_SQUARED) g = m - yy;
            else g = (yy * m < 1.0) ? -yy : 0.0;
            for (int64_t p = row_ptr[t]; p < row_ptr[t + 1]; ++p) w[col[p]] -= eta * g * (val ? (double)val[p] : 1.0);
        }
    return ORC_OK;
}
