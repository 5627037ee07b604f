/*
 * Seeded synthetic sparse examples for serially-equivalent sparse SGD.
 *
 * This file draws INPUTS only: CSR rows of feature ids, their values and the
 * labels.  It contains none of the arithmetic of the method under test (no
 * conflict chains, no levels, no SGD).  Both the CPU oracle and the CUDA path
 * read the arrays it writes.
 *
 * Random numbers: Philox4x32-10, the counter-based generator of Salmon,
 * Moraes, Dror and Shaw, "Parallel random numbers: as easy as 1, 2, 3"
 * (SC'11).  Every row t owns the stream keyed by (seed, purpose tag) with
 * counter (t, draw index), so the output does not depend on the number of
 * threads.
 *
 * Feature-id distributions:
 *   uniform : ids uniform on [0, F), drawn with replacement, duplicates in a
 *             row rejected until k distinct ids are held.
 *   dense   : every example holds features 0 .. k-1 (k <= F; k = F is a
 *             dense matrix).
 *   zipf(s) : rank r in 1..F with probability r^-s / H(F,s), mapped to an id
 *             through one seeded Fisher-Yates permutation of [0, F); the
 *             inverse CDF is evaluated with a guide table (the cutpoint
 *             method of Chen and Asau, 1974) over the fp64 cumulative sums.
 *             Duplicates rejected as above.
 * Each row's ids are stored in ascending order.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    int64_t n_rows, n_cols;
    int32_t k, k_lo;       /* row length uniform in [k_lo, k]; k_lo == k gives fixed length */
    int32_t id_dist;       /* 0 uniform, 1 zipf, 2 dense */
    double zipf_s;
    int32_t val_dist;      /* 0 N(0,1), 1 U(-1,1), 2 all ones */
    int32_t label_kind;    /* 0 sign(w*.x) (sign(0)=+1), 1 Bernoulli(sigmoid(w*.x)) -> +-1, 2 w*.x + noise */
    double wstar_std;      /* w*_j ~ N(0, wstar_std^2) */
    double noise_std;      /* label noise N(0, noise_std^2) for label_kind 2 */
    uint64_t seed, wseed;
    int32_t nthreads;
} synth_cfg;

enum { TAG_LEN = 1, TAG_ID = 2, TAG_VAL = 3, TAG_LABEL = 4, TAG_WSTAR = 5, TAG_PERM = 6 };

/* ---------------------------------------------------------------- Philox */
static void philox4x32_10(const uint32_t ctr[4], uint32_t k0, uint32_t k1, uint32_t out[4])
{
    uint32_t c0 = ctr[0], c1 = ctr[1], c2 = ctr[2], c3 = ctr[3];
    for (int round = 0; round < 10; ++round) {
        uint64_t p0 = (uint64_t)0xD2511F53u * c0;
        uint64_t p1 = (uint64_t)0xCD9E8D57u * c2;
        uint32_t n0 = (uint32_t)(p1 >> 32) ^ c1 ^ k0;
        uint32_t n1 = (uint32_t)p1;
        uint32_t n2 = (uint32_t)(p0 >> 32) ^ c3 ^ k1;
        uint32_t n3 = (uint32_t)p0;
        c0 = n0; c1 = n1; c2 = n2; c3 = n3;
        k0 += 0x9E3779B9u;
        k1 += 0xBB67AE85u;
    }
    out[0] = c0; out[1] = c1; out[2] = c2; out[3] = c3;
}

/* exported for a known-answer check of the generator */
void synth_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4])
{
    philox4x32_10(ctr, key[0], key[1], out);
}

typedef struct {
    uint32_t k0, k1;
    uint64_t stream, idx;
    uint32_t buf[4];
    int avail;
} rng_t;

static void rng_init(rng_t *r, uint64_t seed, uint32_t tag, uint64_t stream)
{
    r->k0 = (uint32_t)seed;
    r->k1 = (uint32_t)(seed >> 32) ^ (tag * 0x9E3779B1u);
    r->stream = stream;
    r->idx = 0;
    r->avail = 0;
}

static uint32_t rng_u32(rng_t *r)
{
    if (r->avail == 0) {
        uint32_t c[4] = {(uint32_t)r->stream, (uint32_t)(r->stream >> 32),
                         (uint32_t)r->idx, (uint32_t)(r->idx >> 32)};
        philox4x32_10(c, r->k0, r->k1, r->buf);
        r->idx++;
        r->avail = 4;
    }
    return r->buf[4 - r->avail--];
}

static uint64_t rng_u64(rng_t *r)
{
    uint64_t hi = rng_u32(r);
    return (hi << 32) | rng_u32(r);
}

/* uniform on [0, 1) with 53 random bits */
static double rng_u01(rng_t *r) { return (double)(rng_u64(r) >> 11) * (1.0 / 9007199254740992.0); }

/* uniform integer on [0, n): multiply-shift of a 64-bit draw (bias <= n / 2^64) */
static uint64_t rng_below(rng_t *r, uint64_t n)
{
    unsigned __int128 m = (unsigned __int128)rng_u64(r) * n;
    return (uint64_t)(m >> 64);
}

/* standard normal by the Box-Muller transform (one of the pair) */
static double rng_normal(rng_t *r)
{
    double u1 = 1.0 - rng_u01(r); /* (0, 1] */
    double u2 = rng_u01(r);
    return sqrt(-2.0 * log(u1)) * cos(6.283185307179586476925 * u2);
}

/* ------------------------------------------------------------ Zipf table */
typedef struct {
    int64_t F;
    double *cdf;     /* cdf[r] = P(rank <= r+1) */
    int64_t *guide;  /* guide[g] = first r with cdf[r] > g/F */
    int32_t *perm;   /* rank -> id */
} zipf_t;

static int zipf_build(zipf_t *z, int64_t F, double s, uint64_t seed)
{
    z->F = F;
    z->cdf = (double *)malloc(sizeof(double) * (size_t)F);
    z->guide = (int64_t *)malloc(sizeof(int64_t) * (size_t)F);
    z->perm = (int32_t *)malloc(sizeof(int32_t) * (size_t)F);
    if (!z->cdf || !z->guide || !z->perm) return -1;
    double acc = 0.0;
    for (int64_t r = 0; r < F; ++r) {
        acc += pow((double)(r + 1), -s);
        z->cdf[r] = acc;
    }
    for (int64_t r = 0; r < F; ++r) z->cdf[r] /= acc;
    z->cdf[F - 1] = 1.0;
    int64_t r = 0;
    for (int64_t g = 0; g < F; ++g) {
        double edge = (double)g / (double)F;
        while (z->cdf[r] <= edge) ++r;
        z->guide[g] = r;
    }
    rng_t pr;
    rng_init(&pr, seed, TAG_PERM, 0);
    for (int64_t i = 0; i < F; ++i) z->perm[i] = (int32_t)i;
    for (int64_t i = F - 1; i > 0; --i) {
        int64_t j = (int64_t)rng_below(&pr, (uint64_t)(i + 1));
        int32_t tmp = z->perm[i];
        z->perm[i] = z->perm[j];
        z->perm[j] = tmp;
    }
    return 0;
}

static void zipf_free(zipf_t *z)
{
    free(z->cdf);
    free(z->guide);
    free(z->perm);
}

static int32_t zipf_draw(const zipf_t *z, rng_t *r)
{
    double u = rng_u01(r);
    int64_t g = (int64_t)(u * (double)z->F);
    if (g >= z->F) g = z->F - 1;
    int64_t rank = z->guide[g];
    while (z->cdf[rank] <= u) ++rank;
    return z->perm[rank];
}

/* ------------------------------------------------------------ row lengths */
static int32_t row_len(const synth_cfg *c, int64_t t)
{
    if (c->k_lo >= c->k) return c->k;
    rng_t r;
    rng_init(&r, c->seed, TAG_LEN, (uint64_t)t);
    return c->k_lo + (int32_t)rng_below(&r, (uint64_t)(c->k - c->k_lo + 1));
}

/* row_ptr[0..n_rows] from the seeded row lengths; returns 0 or -1 on bad config */
int synth_row_ptr(const synth_cfg *c, int64_t *row_ptr)
{
    if (c->n_rows < 0 || c->n_cols <= 0 || c->k < 0 || c->k_lo < 0 || c->k > c->n_cols) return -1;
    row_ptr[0] = 0;
    for (int64_t t = 0; t < c->n_rows; ++t) row_ptr[t + 1] = row_ptr[t] + row_len(c, t);
    return 0;
}

/* ------------------------------------------------------------ rows */
typedef struct {
    const synth_cfg *c;
    const zipf_t *z;
    const float *wstar;
    const int64_t *row_ptr;
    int32_t *col;
    float *val;
    float *y;
    float *wstar_out;
    int64_t lo, hi;     /* rows [lo, hi) or features for the w* pass */
    int status;
} job_t;

static int cmp_i32(const void *a, const void *b)
{
    int32_t x = *(const int32_t *)a, y = *(const int32_t *)b;
    return (x > y) - (x < y);
}

static void *wstar_worker(void *arg)
{
    job_t *j = (job_t *)arg;
    for (int64_t f = j->lo; f < j->hi; ++f) {
        rng_t r;
        rng_init(&r, j->c->wseed, TAG_WSTAR, (uint64_t)f);
        j->wstar_out[f] = (float)(j->c->wstar_std * rng_normal(&r));
    }
    return NULL;
}

static void *row_worker(void *arg)
{
    job_t *j = (job_t *)arg;
    const synth_cfg *c = j->c;
    int cap = 16;
    while (cap < 4 * c->k) cap <<= 1;
    int64_t *set = (int64_t *)malloc(sizeof(int64_t) * (size_t)cap);
    if (!set) { j->status = -2; return NULL; }
    const int64_t max_draws = 100000000;
    for (int64_t t = j->lo; t < j->hi; ++t) {
        int64_t base = j->row_ptr[t];
        int32_t len = (int32_t)(j->row_ptr[t + 1] - base);
        int32_t *ids = j->col + base;
        memset(set, 0, sizeof(int64_t) * (size_t)cap);
        rng_t r;
        rng_init(&r, c->seed, TAG_ID, (uint64_t)t);
        int32_t n = 0;
        int64_t draws = 0;
        while (n < len) {
            if (++draws > max_draws) { j->status = -3; free(set); return NULL; }
            if (c->id_dist == 2) {      /* dense: the example holds features 0 .. len-1 */
                ids[n] = n;
                ++n;
                continue;
            }
            int32_t id = c->id_dist == 1 ? zipf_draw(j->z, &r) : (int32_t)rng_below(&r, (uint64_t)c->n_cols);
            uint64_t h = ((uint64_t)id * 0x9E3779B97F4A7C15ull) >> 20;
            int fresh = 1;
            for (;;) {
                int64_t slot = (int64_t)(h & (uint64_t)(cap - 1));
                if (set[slot] == 0) { set[slot] = (int64_t)id + 1; break; }
                if (set[slot] == (int64_t)id + 1) { fresh = 0; break; }
                ++h;
            }
            if (fresh) ids[n++] = id;
        }
        qsort(ids, (size_t)len, sizeof(int32_t), cmp_i32);
        rng_t rv;
        rng_init(&rv, c->seed, TAG_VAL, (uint64_t)t);
        double margin = 0.0;
        for (int32_t i = 0; i < len; ++i) {
            float v;
            if (c->val_dist == 0) v = (float)rng_normal(&rv);
            else if (c->val_dist == 1) v = (float)(2.0 * rng_u01(&rv) - 1.0);
            else v = 1.0f;
            if (j->val) j->val[base + i] = v;
            margin += (double)j->wstar[ids[i]] * (double)v;
        }
        rng_t rl;
        rng_init(&rl, c->seed, TAG_LABEL, (uint64_t)t);
        float lab;
        if (c->label_kind == 0) lab = margin >= 0.0 ? 1.0f : -1.0f;
        else if (c->label_kind == 1) lab = rng_u01(&rl) < 1.0 / (1.0 + exp(-margin)) ? 1.0f : -1.0f;
        else lab = (float)(margin + c->noise_std * rng_normal(&rl));
        j->y[t] = lab;
    }
    free(set);
    return NULL;
}

static int run_jobs(void *(*fn)(void *), job_t *proto, int64_t total, int nthreads)
{
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    pthread_t th[256];
    job_t jobs[256];
    int64_t chunk = (total + nthreads - 1) / nthreads;
    int started = 0;
    for (int i = 0; i < nthreads; ++i) {
        jobs[i] = *proto;
        jobs[i].lo = (int64_t)i * chunk;
        jobs[i].hi = jobs[i].lo + chunk < total ? jobs[i].lo + chunk : total;
        jobs[i].status = 0;
        if (jobs[i].lo >= jobs[i].hi) continue;
        if (pthread_create(&th[i], NULL, fn, &jobs[i]) != 0) { fn(&jobs[i]); jobs[i].lo = -1; continue; }
        ++started;
    }
    int status = 0;
    for (int i = 0; i < nthreads; ++i) {
        if (jobs[i].lo < 0 || jobs[i].lo >= jobs[i].hi) { if (jobs[i].status) status = jobs[i].status; continue; }
        pthread_join(th[i], NULL);
        if (jobs[i].status) status = jobs[i].status;
    }
    (void)started;
    return status;
}

/* w*[0..F) into wstar (caller-owned) */
int synth_wstar(const synth_cfg *c, float *wstar)
{
    job_t proto;
    memset(&proto, 0, sizeof proto);
    proto.c = c;
    proto.wstar_out = wstar;
    return run_jobs(wstar_worker, &proto, c->n_cols, c->nthreads);
}

/* Fill col/val/y for the rows described by row_ptr.  val may be NULL (ones). */
int synth_fill(const synth_cfg *c, const int64_t *row_ptr, const float *wstar,
               int32_t *col, float *val, float *y)
{
    zipf_t z;
    memset(&z, 0, sizeof z);
    if (c->id_dist == 1 && zipf_build(&z, c->n_cols, c->zipf_s, c->seed) != 0) { zipf_free(&z); return -2; }
    job_t proto;
    memset(&proto, 0, sizeof proto);
    proto.c = c;
    proto.z = &z;
    proto.wstar = wstar;
    proto.row_ptr = row_ptr;
    proto.col = col;
    proto.val = val;
    proto.y = y;
    int st = run_jobs(row_worker, &proto, c->n_rows, c->nthreads);
    if (c->id_dist == 1) zipf_free(&z);
    return st;
}
