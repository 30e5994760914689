/*
 * kvev_oracle.c -- CPU oracle for layer-wise KV-cache eviction.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, obviously correct
 * reference that the GPU library is checked against.  Only the test suite,
 * the smoke check and the benchmark's CPU-baseline leg may load it.  It shares
 * no code, header, table or helper with the CUDA path, and it never calls
 * into it.
 *
 * Everything is computed in double precision on the exact values of the bf16
 * inputs, with plain loops in the order the method states its steps.  The
 * only parallelism is OpenMP over independent (sequence, layer, KV-head)
 * units, which does not change any unit's arithmetic.
 *
 * What the paper fixes and what is a reading:
 *   - Capacity allocation (Sec. 3.3, Eq. 3 and the b_min / rounding rules
 *     that follow it) is stated exactly by the paper.
 *   - The plan (Sec. 3.1, Eq. 1): per layer an operator and a nominal
 *     capacity; FULL means no eviction.
 *   - The retention rules themselves (SnapKV observation-window scoring,
 *     H2O heavy hitters, StreamingLLM sink + recent; Sec. 2.1) are cited, not
 *     defined, by the paper.  They are written here from the published
 *     descriptions of those methods; every detail the paper leaves open is
 *     given one explicit reading, stated in the comment of the function
 *     that applies it.
 *
 * Parity status: allocator, StreamingLLM, identity, kept counts, top-k and
 * pooling are pinned by closed forms, hand cases and brute force; the
 * window-score values are pinned by invariants and closed-form special cases
 * (uniform logits, one dominant key), not by any number printed in the paper
 * (it prints none).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Operator identifiers used by the oracle (its own numbering). */
enum { ORC_FULL = 0, ORC_SNAPKV = 1, ORC_H2O = 2, ORC_STREAMING = 3, ORC_TOVA = 4 };
enum { ORC_POOL_MAX = 0, ORC_POOL_AVG = 1 };
enum { ORC_T_IDENTITY = 0, ORC_T_CAP_Q95 = 1 };

/* ------------------------------------------------------------------------ */
/* bf16 helpers                                                              */
/* ------------------------------------------------------------------------ */

/* Exact value of a bf16 bit pattern (bf16 is the top half of an fp32). */
static double bf16_value(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

static double dot_bf16(const uint16_t *a, const uint16_t *b, int d)
{
    double s = 0.0;
    for (int j = 0; j < d; ++j)
        s += bf16_value(a[j]) * bf16_value(b[j]);
    return s;
}

/* ------------------------------------------------------------------------ */
/* Capacity allocation (Sec. 3.3, Eq. 3)                                     */
/* ------------------------------------------------------------------------ */

static int cmp_double(const void *a, const void *b)
{
    double x = *(const double *)a, y = *(const double *)b;
    return (x > y) - (x < y);
}

/* Across-layer 95th percentile, linear interpolation between order
 * statistics (the usual "type 7" definition). */
double oracle_quantile95(const double *s, int L)
{
    double *v = (double *)malloc(sizeof(double) * (size_t)L);
    memcpy(v, s, sizeof(double) * (size_t)L);
    qsort(v, (size_t)L, sizeof(double), cmp_double);
    double h = 0.95 * (double)(L - 1);
    int lo = (int)floor(h);
    double q = v[lo];
    if (lo + 1 < L)
        q += (h - (double)lo) * (v[lo + 1] - v[lo]);
    free(v);
    return q;
}

/* Largest-remainder rounding of a non-negative real vector whose sum is the
 * integer total: floor every entry, then hand the R = total - sum(floor)
 * leftover units one each to the R largest fractional parts (equal parts go
 * to the lower layer index).  Rounding to nearest and then settling the
 * residual by fractional remainder, as Sec. 3.3 states it, selects the same
 * layers. */
static void largest_remainder(const double *x, int L, int64_t total, int32_t *out)
{
    double *frac = (double *)malloc(sizeof(double) * (size_t)L);
    int64_t sum = 0;
    for (int l = 0; l < L; ++l) {
        double f = floor(x[l]);
        out[l] = (int32_t)f;
        frac[l] = x[l] - f;
        sum += out[l];
    }
    int64_t R = total - sum;
    for (int64_t r = 0; r < R; ++r) {
        int best = -1;
        for (int l = 0; l < L; ++l)
            if (frac[l] >= 0.0 && (best < 0 || frac[l] > frac[best]))
                best = l;
        out[best] += 1;
        frac[best] = -1.0; /* each layer receives at most one unit */
    }
    free(frac);
}

/* Budgets from per-layer scores s[0..L): transform T, shift if the minimum
 * is non-positive, proportional split of B_total (Eq. 3), iterative b_min
 * clamping with proportional redistribution, largest-remainder rounding.
 * Returns 0, or -1 when the request is infeasible (L*b_min > B_total). */
int oracle_alloc_from_scores(int32_t *b_out, const double *s, int L, int64_t B_total,
                             int b_min, int transform)
{
    if (L <= 0 || b_min < 0 || (int64_t)L * b_min > B_total)
        return -1;
    double *t = (double *)malloc(sizeof(double) * (size_t)L);
    double *w = (double *)malloc(sizeof(double) * (size_t)L);
    double *bt = (double *)malloc(sizeof(double) * (size_t)L);
    int *fixed = (int *)calloc((size_t)L, sizeof(int));

    /* T(s): identity (entropy scores) or cap at the 95th percentile (PPL). */
    double cap = transform == ORC_T_CAP_Q95 ? oracle_quantile95(s, L) : 0.0;
    for (int l = 0; l < L; ++l)
        t[l] = transform == ORC_T_CAP_Q95 ? fmin(s[l], cap) : s[l];

    /* Shift by -min + 1e-6 when the transformed minimum is non-positive. */
    double mn = t[0];
    for (int l = 1; l < L; ++l)
        mn = fmin(mn, t[l]);
    if (mn <= 0.0)
        for (int l = 0; l < L; ++l)
            t[l] += -mn + 1e-6;

    /* w_l = T(s_l) / sum_j T(s_j). */
    double tsum = 0.0;
    for (int l = 0; l < L; ++l)
        tsum += t[l];
    for (int l = 0; l < L; ++l)
        w[l] = t[l] / tsum;

    /* Provisional b~_l = B w_l, then fix layers below b_min and re-split the
     * remainder among the others in proportion to their weights, until no
     * further layer drops below b_min. */
    for (;;) {
        int nfixed = 0;
        double wfree = 0.0;
        for (int l = 0; l < L; ++l) {
            if (fixed[l])
                nfixed++;
            else
                wfree += w[l];
        }
        double rest = (double)B_total - (double)nfixed * (double)b_min;
        int changed = 0;
        for (int l = 0; l < L; ++l) {
            if (fixed[l]) {
                bt[l] = (double)b_min;
                continue;
            }
            bt[l] = wfree > 0.0 ? rest * w[l] / wfree : 0.0;
        }
        for (int l = 0; l < L; ++l) {
            if (!fixed[l] && bt[l] < (double)b_min) {
                fixed[l] = 1;
                changed = 1;
            }
        }
        if (!changed)
            break;
    }
    largest_remainder(bt, L, B_total, b_out);
    free(t);
    free(w);
    free(bt);
    free(fixed);
    return 0;
}

/* Budget-sweep rescaling (Sec. 3.3, last rule): scale a completed budget
 * vector to a new total and apply largest-remainder rounding; neither the
 * scores nor the route are recomputed, and no b_min is re-applied. */
int oracle_alloc_rescale(int32_t *b_out, const int32_t *b_in, int L, int64_t B_target)
{
    int64_t sum = 0;
    for (int l = 0; l < L; ++l)
        sum += b_in[l];
    if (L <= 0 || sum <= 0 || B_target < 0)
        return -1;
    double *x = (double *)malloc(sizeof(double) * (size_t)L);
    for (int l = 0; l < L; ++l)
        x[l] = (double)b_in[l] * ((double)B_target / (double)sum);
    largest_remainder(x, L, B_target, b_out);
    free(x);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Observation-window attention scores (SnapKV / H2O prefill rule)           */
/* ------------------------------------------------------------------------ */

/* K: n key rows of d bf16.  Q: G*W window query rows of d bf16, row (g, i)
 * at (g*W + i)*d; query i of the window sits at absolute position
 * t = n - W + i and attends causally to keys 0..t (rows with t < 0 lie before
 * the sequence start and do not exist).  Each row's softmax (scale 1/sqrt(d))
 * runs over all of its visible keys.  The score of key k is the attention it
 * receives summed over the window rows and averaged over the G query heads
 * of the KV group:  raw[k] = (1/G) sum_g sum_i p_{g,i}(k). */
void oracle_window_scores(const uint16_t *K, const uint16_t *Q, int n, int d, int G, int W,
                          double *raw)
{
    double scale = 1.0 / sqrt((double)d);
    double *logit = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    for (int k = 0; k < n; ++k)
        raw[k] = 0.0;
    for (int g = 0; g < G; ++g) {
        for (int i = 0; i < W; ++i) {
            long t = (long)n - W + i;
            if (t < 0)
                continue;
            const uint16_t *q = Q + ((size_t)g * W + i) * (size_t)d;
            double m = -INFINITY;
            for (long k = 0; k <= t; ++k) {
                logit[k] = scale * dot_bf16(q, K + (size_t)k * d, d);
                if (logit[k] > m)
                    m = logit[k];
            }
            double z = 0.0;
            for (long k = 0; k <= t; ++k)
                z += exp(logit[k] - m);
            for (long k = 0; k <= t; ++k)
                raw[k] += exp(logit[k] - m) / z;
        }
    }
    for (int k = 0; k < n; ++k)
        raw[k] /= (double)G;
    free(logit);
}

/* 1-D pooling with stride 1 and same-length output over raw[0..E).  The
 * kernel p is odd; entries outside [0, E) are ignored by max pooling and
 * count as zero for average pooling, which always divides by p. */
void oracle_pool1d(const double *raw, int E, int p, int type, double *out)
{
    int h = p / 2;
    for (int k = 0; k < E; ++k) {
        if (type == ORC_POOL_MAX) {
            double m = -INFINITY;
            for (int j = k - h; j <= k + h; ++j)
                if (j >= 0 && j < E && raw[j] > m)
                    m = raw[j];
            out[k] = m;
        } else {
            double s = 0.0;
            for (int j = k - h; j <= k + h; ++j)
                if (j >= 0 && j < E)
                    s += raw[j];
            out[k] = s / (double)p;
        }
    }
}

/* ------------------------------------------------------------------------ */
/* Selection                                                                 */
/* ------------------------------------------------------------------------ */

typedef struct {
    double key;
    int pos;
} orc_item;

/* Order: larger score first; equal scores keep the lower position first. */
static int cmp_item(const void *a, const void *b)
{
    const orc_item *x = (const orc_item *)a, *y = (const orc_item *)b;
    if (x->key > y->key)
        return -1;
    if (x->key < y->key)
        return 1;
    return (x->pos > y->pos) - (x->pos < y->pos);
}

static int cmp_int(const void *a, const void *b)
{
    int x = *(const int *)a, y = *(const int *)b;
    return (x > y) - (x < y);
}

/* The k positions of [0, E) with the largest keys (ties: lower position),
 * written to out[0..k) in ascending position order. */
void oracle_topk(const double *key, int E, int k, int32_t *out)
{
    orc_item *it = (orc_item *)malloc(sizeof(orc_item) * (size_t)(E > 0 ? E : 1));
    for (int j = 0; j < E; ++j) {
        it[j].key = key[j];
        it[j].pos = j;
    }
    qsort(it, (size_t)E, sizeof(orc_item), cmp_item);
    int *sel = (int *)malloc(sizeof(int) * (size_t)(k > 0 ? k : 1));
    for (int j = 0; j < k; ++j)
        sel[j] = it[j].pos;
    qsort(sel, (size_t)k, sizeof(int), cmp_int);
    for (int j = 0; j < k; ++j)
        out[j] = sel[j];
    free(sel);
    free(it);
}

/* ------------------------------------------------------------------------ */
/* One (sequence, layer, KV-head) unit of prefill eviction                   */
/* ------------------------------------------------------------------------ */

typedef struct {
    int method;       /* ORC_* */
    int n;            /* sequence length */
    int b;            /* nominal capacity of the layer */
    int W;            /* observation window */
    int pool_kernel;  /* SnapKV pooling width (odd) */
    int pool_type;    /* ORC_POOL_MAX / ORC_POOL_AVG */
    int sink;         /* StreamingLLM sink tokens */
    int recent;       /* StreamingLLM recent tokens, -1: b - sink */
    int h2o_recent;   /* H2O recent window, -1: floor(b/2) */
    const uint16_t *K; /* [n][d] bf16 bits */
    const uint16_t *Q; /* [G][W][d] bf16 bits (SnapKV / H2O) */
    double *raw;      /* out [n]: window scores (scoring rules), may be NULL */
    double *pooled;   /* out [n]: SnapKV pooled prefix scores, may be NULL */
    int32_t *idx;     /* out [b]: kept positions ascending, padded with -1 */
    int32_t *count;   /* out: number of kept positions */
    double *acc;      /* out [b]: H2O initial accumulated attention, may be NULL */
} oracle_unit;

static void keep_range(int32_t *idx, int *m, int lo, int hi)
{
    for (int p = lo; p < hi; ++p)
        idx[(*m)++] = p;
}

/* Returns 0, or -1 on a parameter the rule cannot accept. */
int oracle_evict_unit(oracle_unit *u, int d, int G)
{
    int n = u->n, b = u->b, m = 0;
    for (int j = 0; j < b; ++j)
        u->idx[j] = -1;
    if (u->acc)
        for (int j = 0; j < b; ++j)
            u->acc[j] = 0.0;

    switch (u->method) {
    case ORC_FULL:
        /* No eviction in this phase: every position stays. */
        *u->count = n;
        return 0;

    case ORC_STREAMING: {
        if (b <= u->sink)
            return -1;
        int recent = u->recent < 0 ? b - u->sink : (u->recent < b - u->sink ? u->recent : b - u->sink);
        int cap = u->sink + recent;
        if (n <= cap) {
            keep_range(u->idx, &m, 0, n);
        } else {
            keep_range(u->idx, &m, 0, u->sink);
            keep_range(u->idx, &m, n - recent, n);
        }
        *u->count = m;
        return 0;
    }

    case ORC_SNAPKV: {
        if (b <= u->W || u->pool_kernel < 1 || (u->pool_kernel & 1) == 0)
            return -1;
        if (u->raw)
            oracle_window_scores(u->K, u->Q, n, d, G, u->W, u->raw);
        if (n <= b) {
            keep_range(u->idx, &m, 0, n);
            *u->count = m;
            return 0;
        }
        int E = n - u->W; /* prefix outside the window */
        double *raw = u->raw ? u->raw : (double *)malloc(sizeof(double) * (size_t)n);
        if (!u->raw)
            oracle_window_scores(u->K, u->Q, n, d, G, u->W, raw);
        double *pooled = u->pooled ? u->pooled : (double *)malloc(sizeof(double) * (size_t)E);
        oracle_pool1d(raw, E, u->pool_kernel, u->pool_type, pooled);
        oracle_topk(pooled, E, b - u->W, u->idx);
        m = b - u->W;
        keep_range(u->idx, &m, E, n); /* the window itself is always kept */
        *u->count = m;
        if (!u->raw)
            free(raw);
        if (!u->pooled)
            free(pooled);
        return 0;
    }

    case ORC_H2O: {
        int r = u->h2o_recent < 0 ? b / 2 : u->h2o_recent;
        if (b < 1 || r > b)
            return -1;
        double *raw = u->raw ? u->raw : (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
        oracle_window_scores(u->K, u->Q, n, d, G, u->W, raw);
        if (n <= b) {
            keep_range(u->idx, &m, 0, n);
        } else {
            int E = n - r;
            oracle_topk(raw, E, b - r, u->idx);
            m = b - r;
            keep_range(u->idx, &m, E, n); /* recent window */
        }
        *u->count = m;
        /* The kept tokens' scores seed the accumulated-attention state. */
        if (u->acc)
            for (int j = 0; j < m; ++j)
                u->acc[j] = raw[u->idx[j]];
        if (!u->raw)
            free(raw);
        return 0;
    }
    default:
        return -1;
    }
}

/* Run many independent units; returns the number of units that failed. */
int oracle_evict_units(oracle_unit *units, int num_units, int d, int G, int nthreads)
{
    int failed = 0;
#ifdef _OPENMP
    if (nthreads > 0)
        omp_set_num_threads(nthreads);
#else
    (void)nthreads;
#endif
#pragma omp parallel for schedule(dynamic, 1) reduction(+ : failed)
    for (int i = 0; i < num_units; ++i)
        failed += oracle_evict_unit(&units[i], d, G) != 0;
    return failed;
}

int oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ------------------------------------------------------------------------ */
/* Decode-phase update of one unit (one generated token)                     */
/* ------------------------------------------------------------------------ */

/* Slots form a set keyed by position; slot order carries no meaning. */
typedef struct {
    int method;      /* ORC_* (decode-phase operator of the layer) */
    int b;           /* nominal capacity */
    int sink, recent;   /* StreamingLLM */
    int h2o_recent;     /* H2O recent window, -1: floor(b/2) */
    int n;           /* sequence length before this step; new token is at position n */
    int cap;         /* slot capacity of the arrays */
    int count;       /* in/out: occupied slots */
    int32_t *pos;    /* [cap] */
    double *acc;     /* [cap] accumulated attention (H2O) */
    uint16_t *K;     /* [cap][d] */
    uint16_t *V;     /* [cap][d] */
    const uint16_t *k_new; /* [d] */
    const uint16_t *v_new; /* [d] */
    const uint16_t *q_new; /* [G][d] query of the new token, one row per head of the group */
    int evicted;     /* out: evicted position, -1 if none */
} oracle_dec_unit;

static void remove_slot(oracle_dec_unit *u, int j, int d)
{
    int last = u->count - 1;
    if (j != last) {
        u->pos[j] = u->pos[last];
        u->acc[j] = u->acc[last];
        memcpy(u->K + (size_t)j * d, u->K + (size_t)last * d, sizeof(uint16_t) * (size_t)d);
        memcpy(u->V + (size_t)j * d, u->V + (size_t)last * d, sizeof(uint16_t) * (size_t)d);
    }
    u->count = last;
}

/* Attention of the new token's G query rows over every current slot
 * (the new token included), averaged over the group: p[j] = (1/G) sum_g
 * softmax_j(q_g . K_j / sqrt(d)). */
static void decode_attention(const oracle_dec_unit *u, int d, int G, double *p)
{
    double scale = 1.0 / sqrt((double)d);
    double *lg = (double *)malloc(sizeof(double) * (size_t)u->count);
    for (int j = 0; j < u->count; ++j)
        p[j] = 0.0;
    for (int g = 0; g < G; ++g) {
        const uint16_t *q = u->q_new + (size_t)g * d;
        double m = -INFINITY;
        for (int j = 0; j < u->count; ++j) {
            lg[j] = scale * dot_bf16(q, u->K + (size_t)j * d, d);
            if (lg[j] > m)
                m = lg[j];
        }
        double z = 0.0;
        for (int j = 0; j < u->count; ++j)
            z += exp(lg[j] - m);
        for (int j = 0; j < u->count; ++j)
            p[j] += exp(lg[j] - m) / z;
    }
    for (int j = 0; j < u->count; ++j)
        p[j] /= (double)G;
    free(lg);
}

int oracle_decode_unit(oracle_dec_unit *u, int d, int G)
{
    u->evicted = -1;
    if (u->count >= u->cap)
        return -1;
    /* 1. Append the new token. */
    int j0 = u->count++;
    u->pos[j0] = u->n;
    u->acc[j0] = 0.0;
    memcpy(u->K + (size_t)j0 * d, u->k_new, sizeof(uint16_t) * (size_t)d);
    memcpy(u->V + (size_t)j0 * d, u->v_new, sizeof(uint16_t) * (size_t)d);
    int newlen = u->n + 1;

    if (u->method == ORC_H2O || u->method == ORC_TOVA) {
        double *p = (double *)malloc(sizeof(double) * (size_t)u->count);
        decode_attention(u, d, G, p);
        /* H2O accumulates; TOVA keeps only the current step's attention. */
        for (int j = 0; j < u->count; ++j)
            u->acc[j] = u->method == ORC_H2O ? u->acc[j] + p[j] : p[j];
        free(p);
        if (u->count > u->b) {
            int r = u->method == ORC_H2O ? (u->h2o_recent < 0 ? u->b / 2 : u->h2o_recent) : 0;
            int limit = newlen - r; /* positions >= limit form the protected recent window */
            int best = -1;
            for (int j = 0; j < u->count; ++j) {
                if (u->pos[j] >= limit)
                    continue;
                if (best < 0 || u->acc[j] < u->acc[best] ||
                    (u->acc[j] == u->acc[best] && u->pos[j] > u->pos[best]))
                    best = j;
            }
            if (best < 0)
                return -1;
            u->evicted = u->pos[best];
            remove_slot(u, best, d);
        }
    } else if (u->method == ORC_STREAMING) {
        int recent = u->recent < 0 ? u->b - u->sink
                                   : (u->recent < u->b - u->sink ? u->recent : u->b - u->sink);
        if (u->count > u->sink + recent) {
            int best = -1;
            for (int j = 0; j < u->count; ++j)
                if (u->pos[j] >= u->sink && (best < 0 || u->pos[j] < u->pos[best]))
                    best = j;
            u->evicted = u->pos[best];
            remove_slot(u, best, d);
        }
    }
    /* SnapKV and FULL have no decode-phase eviction: append only. */
    u->n = newlen;
    return 0;
}

int oracle_decode_units(oracle_dec_unit *units, int num_units, int d, int G, int nthreads)
{
    int failed = 0;
#ifdef _OPENMP
    if (nthreads > 0)
        omp_set_num_threads(nthreads);
#else
    (void)nthreads;
#endif
#pragma omp parallel for schedule(dynamic, 1) reduction(+ : failed)
    for (int i = 0; i < num_units; ++i)
        failed += oracle_decode_unit(&units[i], d, G) != 0;
    return failed;
}
