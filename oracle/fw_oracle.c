/*
 * fw_oracle.c -- plain, slow, fp64 CPU oracle for forced-weight subset
 * evaluation ("Trust the Mass: Forced Weights in KV-Cache Eviction").
 *
 * TEST INFRASTRUCTURE.  Only tests/, __graft_entry__.smoke() and bench.py's
 * CPU-baseline / reference legs load this library.  It shares no code, header,
 * table or helper with the CUDA library; it is written from the paper's
 * definitions, in the paper's order, with no blocking or fusion:
 *
 *   Definition 2.1 (instance, kept set A, p(A), dropped mass 1 - p(A), m_A,
 *                   top-mass set A*_s, D)
 *   Sec. 2.1        es(A) = ||mu - m_A||, ES(s) = min_{|A|=s} es(A)
 *   Lemma 2.1       es(A) = pbar(A)||m_{A^c} - m_A|| = ||g_A|| / p(A)
 *   Sec. 2.1        balancing selector: from A*_s, repeatedly take the one
 *                   kept<->dropped swap that most decreases es(A); stop when
 *                   none decreases it
 *   Definition 2.2  candidate set = top-mass set + keys of largest single-key
 *                   error p_j ||v_j - mu||
 *   Definition 2.2  ES_pool: exact minimum of es over the size-s subsets of
 *                   the candidate set
 *   Sec. 2.1        group vote: one kept set per KV head, the s keys of
 *                   largest mass summed over the head's query rows, scored
 *                   for every row of the group
 *   Sec. 4          ContourKV: one score r, one global threshold tau, a
 *                   recency floor of the last 32 positions per cell, tau set
 *                   so that the cache averages s entries per cell; ragged
 *                   per-head storage that frees the evicted bytes
 *
 * Readings taken where the paper is silent:
 *   - p is the softmax of the fp32 logits computed in fp64 (std exp);
 *   - top-mass ranks by logit, equal logits -> lower index first; -0 == +0;
 *   - dropped mass is summed over the dropped keys, not formed as 1 - p(A);
 *   - swap pool: removal from every kept key, addition from the E dropped
 *     keys of largest single-key error (ties -> lower index); swapped-out keys
 *     stay in the pool; the most-decreasing pair wins, ties -> smallest
 *     (i, j) lexicographically; a swap is taken only on a strict decrease;
 *   - best subset: exact ties -> smallest colex rank sum_i C(c_i, i);
 *   - group vote: equal summed mass -> lower index first;
 *   - ContourKV: ties at tau are broken by (score desc, cell asc, pos asc);
 *     floor = last min(32, T) positions; the per-cell dropped mass is that of
 *     the cell's normalised scores, for the allocated set and for the cell's
 *     own top-s set (s = average budget).
 *
 * Build: gcc -O2 -fopenmp -fPIC -shared fw_oracle.c -lm
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORC_OK 0
#define ORC_ERR_ARG 1
#define ORC_ERR_NONFINITE 6

/* A batch of attention rows.  Rows come in groups of rows_per_group rows that
 * share one value block and one length n[g] (a KV head, a GQA group, or a
 * single row).  Row r = g * rows_per_group + i has logits at
 * logits + logit_off[g] + i * n[g] and values V_g = v + v_off[g] (n[g] x d,
 * row-major).  v_dtype: 0 = float32, 1 = bfloat16 bit patterns, 2 = float64. */
typedef struct {
    int64_t num_groups;
    int32_t rows_per_group;
    int32_t d;
    const float *logits;
    const int64_t *logit_off;
    const int32_t *n;
    const void *v;
    const int64_t *v_off;
    int32_t v_dtype;
} orc_rows;

/* ---------------------------------------------------------------- helpers */

static double v_at(const orc_rows *R, int64_t off)
{
    if (R->v_dtype == 0)
        return (double)((const float *)R->v)[off];
    if (R->v_dtype == 1) {
        uint32_t bits = ((uint32_t)((const uint16_t *)R->v)[off]) << 16;
        float f;
        memcpy(&f, &bits, sizeof f);
        return (double)f;
    }
    return ((const double *)R->v)[off];
}

/* One instance (Definition 2.1): masses p (length n) and points v (n x d). */
typedef struct {
    int n, d;
    double *p;   /* [n] */
    double *v;   /* [n][d] */
    double *mu;  /* [d] dense output mu = sum_j p_j v_j */
    const float *logit; /* [n] */
} instance;

static void instance_free(instance *I)
{
    free(I->p);
    free(I->v);
    free(I->mu);
}

/* softmax in fp64: p_j = exp(l_j - M) / sum_i exp(l_i - M), M = max_i l_i.
 * Returns 0, or ORC_ERR_NONFINITE if any logit is not finite. */
static int softmax_f64(int n, const float *l, double *p)
{
    double M = -INFINITY, Z = 0.0;
    for (int j = 0; j < n; ++j) {
        if (!isfinite(l[j]))
            return ORC_ERR_NONFINITE;
        if ((double)l[j] > M)
            M = (double)l[j];
    }
    for (int j = 0; j < n; ++j) {
        p[j] = exp((double)l[j] - M);
        Z += p[j];
    }
    for (int j = 0; j < n; ++j)
        p[j] /= Z;
    return 0;
}

static void dense_output(instance *I)
{
    for (int c = 0; c < I->d; ++c)
        I->mu[c] = 0.0;
    for (int j = 0; j < I->n; ++j)
        for (int c = 0; c < I->d; ++c)
            I->mu[c] += I->p[j] * I->v[(int64_t)j * I->d + c];
}

/* Build instance for row r of batch R.  Returns status. */
static int load_row(const orc_rows *R, int64_t r, instance *I)
{
    int64_t g = r / R->rows_per_group;
    int64_t i = r % R->rows_per_group;
    int n = R->n[g], d = R->d;
    I->n = n;
    I->d = d;
    I->logit = R->logits + R->logit_off[g] + i * (int64_t)n;
    I->p = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    I->v = (double *)malloc(sizeof(double) * (size_t)n * (size_t)d + 8);
    I->mu = (double *)malloc(sizeof(double) * (size_t)d);
    for (int64_t e = 0; e < (int64_t)n * d; ++e)
        I->v[e] = v_at(R, R->v_off[g] + e);
    int st = softmax_f64(n, I->logit, I->p);
    if (st)
        return st;
    dense_output(I);
    return 0;
}

typedef struct {
    double key;
    int idx;
} keyed;

/* larger key first; equal keys -> lower index first */
static int cmp_desc_key_asc_idx(const void *a, const void *b)
{
    const keyed *x = (const keyed *)a, *y = (const keyed *)b;
    if (x->key > y->key) return -1;
    if (x->key < y->key) return 1;
    return (x->idx > y->idx) - (x->idx < y->idx);
}

/* Top-mass set by logit (Definition 2.1, tie reading: lower index first):
 * in_A[j] = 1 for the first k of the order (logit desc, index asc). */
static void topk_by_logit(int n, const float *l, int k, unsigned char *in_A)
{
    if (n < 1)
        return;
    keyed *o = (keyed *)malloc(sizeof(keyed) * (size_t)(n > 0 ? n : 1));
    for (int j = 0; j < n; ++j) {
        o[j].key = (double)l[j]; /* -0.0 and +0.0 compare equal as doubles */
        o[j].idx = j;
    }
    qsort(o, (size_t)n, sizeof(keyed), cmp_desc_key_asc_idx);
    memset(in_A, 0, (size_t)n);
    for (int t = 0; t < k && t < n; ++t)
        in_A[o[t].idx] = 1;
    free(o);
}

/* Everything Definition 2.1 / Lemma 2.1 say about one kept set A. */
typedef struct {
    double kept_mass;  /* p(A) = sum_{j in A} p_j                          */
    double dropped;    /* sum_{j not in A} p_j  (= 1 - p(A))               */
    double gap;        /* es(A) = ||m_A - mu||                             */
    double phi;        /* ||g_A||, g_A = sum_{j in A} p_j (v_j - mu)       */
    double form1;      /* pbar(A) ||m_{A^c} - m_A||   (Lemma 2.1)          */
    double form2;      /* ||g_A|| / p(A)              (Lemma 2.1)          */
} set_eval;

/* m_A written to mA (may be NULL). */
static set_eval eval_set(const instance *I, const unsigned char *in_A, double *mA)
{
    int n = I->n, d = I->d;
    set_eval e;
    double *NA = (double *)calloc((size_t)d, sizeof(double));
    double *NC = (double *)calloc((size_t)d, sizeof(double));
    double *gA = (double *)calloc((size_t)d, sizeof(double));
    double PA = 0.0, PC = 0.0;
    for (int j = 0; j < n; ++j) {
        const double *vj = I->v + (int64_t)j * d;
        if (in_A[j]) {
            PA += I->p[j];
            for (int c = 0; c < d; ++c) {
                NA[c] += I->p[j] * vj[c];
                gA[c] += I->p[j] * (vj[c] - I->mu[c]);
            }
        } else {
            PC += I->p[j];
            for (int c = 0; c < d; ++c)
                NC[c] += I->p[j] * vj[c];
        }
    }
    double gap2 = 0.0, f1 = 0.0, phi2 = 0.0;
    for (int c = 0; c < d; ++c) {
        double m_A = PA > 0 ? NA[c] / PA : 0.0;
        double m_C = PC > 0 ? NC[c] / PC : 0.0;
        if (mA)
            mA[c] = m_A;
        gap2 += (m_A - I->mu[c]) * (m_A - I->mu[c]);
        f1 += (m_C - m_A) * (m_C - m_A);
        phi2 += gA[c] * gA[c];
    }
    e.kept_mass = PA;
    e.dropped = PC;
    e.gap = sqrt(gap2);
    e.phi = sqrt(phi2);
    e.form1 = PC > 0 ? PC * sqrt(f1) : 0.0;
    e.form2 = PA > 0 ? e.phi / PA : 0.0;
    free(NA);
    free(NC);
    free(gA);
    return e;
}

/* es(A) of the set given by its members, straight from the definition. */
static double es_of_members(const instance *I, const int *members, int k, double *NA)
{
    int d = I->d;
    double PA = 0.0, gap2 = 0.0;
    for (int c = 0; c < d; ++c)
        NA[c] = 0.0;
    for (int t = 0; t < k; ++t) {
        int j = members[t];
        PA += I->p[j];
        for (int c = 0; c < d; ++c)
            NA[c] += I->p[j] * I->v[(int64_t)j * d + c];
    }
    for (int c = 0; c < d; ++c) {
        double diff = NA[c] / PA - I->mu[c];
        gap2 += diff * diff;
    }
    return sqrt(gap2);
}

/* ------------------------------------------------------------ public API */

/* Single instance given directly by masses (Definition 2.1, no softmax) and a
 * kept set mask.  Outputs mu[d], mA[d] and the set_eval fields
 * out6 = {p(A), dropped, es, ||g_A||, form1, form2}. */
int orc_eval_instance(int n, int d, const double *p, const double *v,
                      const unsigned char *in_A, double *mu, double *mA, double *out6)
{
    if (n < 1 || d < 1)
        return ORC_ERR_ARG;
    instance I;
    I.n = n;
    I.d = d;
    I.p = (double *)p;
    I.v = (double *)v;
    I.mu = mu;
    I.logit = NULL;
    dense_output(&I);
    set_eval e = eval_set(&I, in_A, mA);
    out6[0] = e.kept_mass;
    out6[1] = e.dropped;
    out6[2] = e.gap;
    out6[3] = e.phi;
    out6[4] = e.form1;
    out6[5] = e.form2;
    return ORC_OK;
}

/* a1-a4: softmax, dense output, top-k kept sets, forced-weight outputs, gap,
 * dropped mass, ||g_A|| and the two Lemma 2.1 forms, per row and budget.
 * k: [rows][nb].  Outputs (any may be NULL):
 *   o [rows][d], o_kept [rows][nb][d], gap/dropped/kept_mass/phi/form1/form2
 *   [rows][nb], kept_bits [rows][nb][words] (bit j of word j/32 = j in A),
 *   status [rows]. */
int orc_dense_and_topk_gap(const orc_rows *R, int nb, const int32_t *k,
                           double *o, double *o_kept, double *gap, double *dropped,
                           double *kept_mass, double *phi, double *form1, double *form2,
                           uint32_t *kept_bits, int words, int32_t *status)
{
    int64_t rows = R->num_groups * R->rows_per_group;
    int d = R->d;
    int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad)
    for (int64_t r = 0; r < rows; ++r) {
        instance I;
        int st = load_row(R, r, &I);
        if (status)
            status[r] = st;
        if (st) {
            instance_free(&I);
            continue;
        }
        if (o)
            for (int c = 0; c < d; ++c)
                o[r * d + c] = I.mu[c];
        unsigned char *in_A = (unsigned char *)malloc((size_t)I.n + 1);
        for (int b = 0; b < nb; ++b) {
            int kb = k[r * nb + b];
            if (kb < 1 || kb > I.n) {
                bad |= 1;
                continue;
            }
            topk_by_logit(I.n, I.logit, kb, in_A);
            double *mA = o_kept ? o_kept + (r * nb + b) * (int64_t)d : NULL;
            set_eval e = eval_set(&I, in_A, mA);
            int64_t rb = r * nb + b;
            if (gap) gap[rb] = e.gap;
            if (dropped) dropped[rb] = e.dropped;
            if (kept_mass) kept_mass[rb] = e.kept_mass;
            if (phi) phi[rb] = e.phi;
            if (form1) form1[rb] = e.form1;
            if (form2) form2[rb] = e.form2;
            if (kept_bits) {
                uint32_t *w = kept_bits + rb * (int64_t)words;
                for (int t = 0; t < words; ++t)
                    w[t] = 0u;
                for (int j = 0; j < I.n; ++j)
                    if (in_A[j])
                        w[j >> 5] |= 1u << (j & 31);
            }
        }
        free(in_A);
        instance_free(&I);
    }
    return bad ? ORC_ERR_ARG : ORC_OK;
}

/* a5: the balancing selector (Sec. 2.1) inside the candidate set of
 * Definition 2.2.  Per row and budget:
 *   A <- top-mass set A*_k; X <- the E dropped keys of largest p_j||v_j - mu||
 *   (ties -> lower index); pool = A u X.
 *   repeat: evaluate es(A - i + j) for every i in A, j in pool \ A (from the
 *   definition: m_A' = N_A' / p(A')); take the minimum (ties -> smallest
 *   (i, j)); accept it iff it is strictly below es(A); stop otherwise or after
 *   max_swaps swaps.
 * Outputs: n_swaps [rows][nb]; swap_out/swap_in [rows][nb][max_swaps] (in the
 * order taken); refined_gap, topk_gap [rows][nb]; capped [rows][nb];
 * margin [rows][nb] = the smallest decision margin over all rounds, relative
 * to the round's starting es: min((runner-up - best)/es, |es - best|/es);
 * pool_margin [rows][nb] = (e_E - e_{E+1}) / e_E for the single-key errors at
 * the pool boundary (+inf when every dropped key is in the pool). */
int orc_swap_refine(const orc_rows *R, int nb, const int32_t *k, int E, int max_swaps,
                    int32_t *n_swaps, int32_t *swap_out, int32_t *swap_in,
                    double *refined_gap, double *topk_gap, int32_t *capped,
                    double *margin, double *pool_margin)
{
    int64_t rows = R->num_groups * R->rows_per_group;
    int d = R->d;
    int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad)
    for (int64_t r = 0; r < rows; ++r) {
        instance I;
        if (load_row(R, r, &I)) {
            instance_free(&I);
            bad |= 2;
            continue;
        }
        int n = I.n;
        unsigned char *in_A = (unsigned char *)malloc((size_t)n + 1);
        unsigned char *in_pool = (unsigned char *)malloc((size_t)n + 1);
        keyed *err = (keyed *)malloc(sizeof(keyed) * (size_t)n);
        double *NA = (double *)malloc(sizeof(double) * (size_t)d);
        int *kept_list = (int *)malloc(sizeof(int) * (size_t)n);
        int *add_list = (int *)malloc(sizeof(int) * (size_t)n);
        for (int b = 0; b < nb; ++b) {
            int64_t rb = r * nb + b;
            int kb = k[rb];
            if (kb < 1 || kb > n) {
                bad |= 1;
                continue;
            }
            topk_by_logit(n, I.logit, kb, in_A);
            /* candidate set: single-key errors of the dropped keys */
            int nd = 0;
            for (int j = 0; j < n; ++j) {
                if (in_A[j])
                    continue;
                double s = 0.0;
                for (int c = 0; c < d; ++c) {
                    double t = I.v[(int64_t)j * d + c] - I.mu[c];
                    s += t * t;
                }
                err[nd].key = I.p[j] * sqrt(s);
                err[nd].idx = j;
                ++nd;
            }
            qsort(err, (size_t)nd, sizeof(keyed), cmp_desc_key_asc_idx);
            int Eeff = E < nd ? E : nd;
            memcpy(in_pool, in_A, (size_t)n);
            for (int t = 0; t < Eeff; ++t)
                in_pool[err[t].idx] = 1;
            if (pool_margin)
                pool_margin[rb] = (Eeff < nd && Eeff > 0)
                                      ? (err[Eeff - 1].key - err[Eeff].key) / err[Eeff - 1].key
                                      : INFINITY;
            /* greedy best-improvement swaps */
            double cur = eval_set(&I, in_A, NULL).gap;
            if (topk_gap)
                topk_gap[rb] = cur;
            double min_margin = INFINITY;
            int taken = 0, cap = 0;
            for (;;) {
                /* N_A and p(A) of the current set */
                double PA = 0.0;
                for (int c = 0; c < d; ++c)
                    NA[c] = 0.0;
                for (int j = 0; j < n; ++j)
                    if (in_A[j]) {
                        PA += I.p[j];
                        for (int c = 0; c < d; ++c)
                            NA[c] += I.p[j] * I.v[(int64_t)j * d + c];
                    }
                double best = INFINITY, second = INFINITY;
                int bi = -1, bj = -1;
                int na = 0, nadd = 0;
                for (int j = 0; j < n; ++j) {
                    if (in_A[j])
                        kept_list[na++] = j;
                    else if (in_pool[j])
                        add_list[nadd++] = j;
                }
                for (int a = 0; a < na; ++a) {
                    int i = kept_list[a];
                    for (int q = 0; q < nadd; ++q) {
                        int j = add_list[q];
                        double P2 = PA - I.p[i] + I.p[j];
                        double g2 = 0.0;
                        for (int c = 0; c < d; ++c) {
                            double Nc = NA[c] - I.p[i] * I.v[(int64_t)i * d + c] +
                                        I.p[j] * I.v[(int64_t)j * d + c];
                            double diff = Nc / P2 - I.mu[c];
                            g2 += diff * diff;
                        }
                        double es_ij = sqrt(g2);
                        if (es_ij < best) {
                            second = best;
                            best = es_ij;
                            bi = i;
                            bj = j;
                        } else if (es_ij < second) {
                            second = es_ij;
                        }
                    }
                }
                if (bi < 0)
                    break; /* no pair exists (k = n or empty pool) */
                if (cur > 0.0) {
                    double m1 = (second - best) / cur;
                    double m2 = fabs(cur - best) / cur;
                    double m = m1 < m2 ? m1 : m2;
                    if (m < min_margin)
                        min_margin = m;
                }
                if (!(best < cur))
                    break;
                if (taken >= max_swaps) {
                    cap = 1;
                    break;
                }
                in_A[bi] = 0;
                in_A[bj] = 1;
                if (swap_out)
                    swap_out[rb * max_swaps + taken] = bi;
                if (swap_in)
                    swap_in[rb * max_swaps + taken] = bj;
                ++taken;
                cur = eval_set(&I, in_A, NULL).gap;
            }
            if (n_swaps) n_swaps[rb] = taken;
            if (refined_gap) refined_gap[rb] = cur;
            if (capped) capped[rb] = cap;
            if (margin) margin[rb] = min_margin;
        }
        free(in_A);
        free(in_pool);
        free(err);
        free(NA);
        free(kept_list);
        free(add_list);
        instance_free(&I);
    }
    return bad ? ORC_ERR_ARG : ORC_OK;
}

/* binomial coefficient C(a, b) as uint64 (0 when b > a) */
static uint64_t binom(int a, int b)
{
    if (b < 0 || b > a)
        return 0;
    uint64_t r = 1;
    for (int t = 1; t <= b; ++t)
        r = r * (uint64_t)(a - b + t) / (uint64_t)t;
    return r;
}

/* colex rank of an ascending combination c_1 < ... < c_k (0-based values):
 * sum_{i=1..k} C(c_i, i). */
uint64_t orc_colex_rank(int k, const int32_t *c)
{
    uint64_t r = 0;
    for (int i = 0; i < k; ++i)
        r += binom(c[i], i + 1);
    return r;
}

/* a6: ES(k) = min over all size-k subsets of es(A) (Sec. 2.1), by exhaustive
 * enumeration in lexicographic order, es from scratch for each subset.
 * Ties in the minimum -> smallest colex rank.  Outputs per row:
 *   best_rank (colex), best_gap, best_idx [rows][k], second_gap (smallest es
 *   among all other subsets; +inf if C(n,k) = 1), topk_gap.  n <= 40. */
int orc_best_subset(const orc_rows *R, const int32_t *k, uint64_t *best_rank,
                    double *best_gap, int32_t *best_idx, int kmax, double *second_gap,
                    double *topk_gap)
{
    int64_t rows = R->num_groups * R->rows_per_group;
    int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad)
    for (int64_t r = 0; r < rows; ++r) {
        instance I;
        if (load_row(R, r, &I)) {
            instance_free(&I);
            bad |= 2;
            continue;
        }
        int n = I.n, kk = k[r];
        if (kk < 1 || kk > n || n > 40 || kk > kmax) {
            instance_free(&I);
            bad |= 1;
            continue;
        }
        if (topk_gap) {
            unsigned char *in_A = (unsigned char *)malloc((size_t)n);
            topk_by_logit(n, I.logit, kk, in_A);
            topk_gap[r] = eval_set(&I, in_A, NULL).gap;
            free(in_A);
        }
        int c[64], bestc[64];
        double *scratch = (double *)malloc(sizeof(double) * (size_t)R->d);
        for (int i = 0; i < kk; ++i)
            c[i] = i;
        double best = INFINITY, second = INFINITY;
        uint64_t brank = 0;
        for (;;) {
            double es = es_of_members(&I, c, kk, scratch);
            uint64_t rank = orc_colex_rank(kk, c);
            if (es < best || (es == best && rank < brank)) {
                if (best < second)
                    second = best;
                best = es;
                brank = rank;
                memcpy(bestc, c, sizeof(int) * (size_t)kk);
            } else if (es < second) {
                second = es;
            }
            /* next combination in lexicographic order */
            int i = kk - 1;
            while (i >= 0 && c[i] == n - kk + i)
                --i;
            if (i < 0)
                break;
            ++c[i];
            for (int t = i + 1; t < kk; ++t)
                c[t] = c[t - 1] + 1;
        }
        if (best_rank) best_rank[r] = brank;
        if (best_gap) best_gap[r] = best;
        if (second_gap) second_gap[r] = second;
        if (best_idx)
            for (int i = 0; i < kk; ++i)
                best_idx[r * kmax + i] = bestc[i];
        free(scratch);
        instance_free(&I);
    }
    return bad ? ORC_ERR_ARG : ORC_OK;
}

/* ---------------------------------------------------------- ContourKV */

typedef struct {
    double score;
    int cell;
    int pos;
} cand;

/* score desc, then cell asc, then position asc */
static int cmp_cand(const void *a, const void *b)
{
    const cand *x = (const cand *)a, *y = (const cand *)b;
    if (x->score > y->score) return -1;
    if (x->score < y->score) return 1;
    if (x->cell != y->cell) return x->cell < y->cell ? -1 : 1;
    return (x->pos > y->pos) - (x->pos < y->pos);
}

/* a7: ContourKV allocation (Sec. 4).  scores [cells][T] fp32.  Each cell keeps
 * the recency floor F (last min(floor, T) positions) plus every non-floor
 * position among the K = total_budget - sum |F| best non-floor entries of the
 * whole cache under (score desc, cell asc, pos asc); tau = score of the K-th.
 * Outputs: counts [cells], offsets [cells+1] (exclusive prefix sum),
 * kept_pos [total_budget] (per cell ascending), tau, dropped_uniform [cells]
 * and dropped_alloc [cells] (mass of the cell's normalised scores outside the
 * kept set: the cell's own top-uniform_s set, and the allocated set). */
int orc_contour_alloc(const float *scores, int cells, int T, int floor_, int64_t total_budget,
                      int uniform_s, int32_t *counts, int64_t *offsets, int32_t *kept_pos,
                      float *tau, double *dropped_uniform, double *dropped_alloc)
{
    if (cells < 1 || T < 1 || floor_ < 0)
        return ORC_ERR_ARG;
    int F = floor_ < T ? floor_ : T;
    int64_t nfloor = (int64_t)cells * F;
    if (total_budget < nfloor || total_budget > (int64_t)cells * T)
        return ORC_ERR_ARG;
    for (int64_t e = 0; e < (int64_t)cells * T; ++e)
        if (!isfinite(scores[e]))
            return ORC_ERR_NONFINITE;
    int64_t nc = (int64_t)cells * (T - F);
    cand *all = (cand *)malloc(sizeof(cand) * (size_t)(nc > 0 ? nc : 1));
    int64_t t = 0;
    for (int h = 0; h < cells; ++h)
        for (int j = 0; j < T - F; ++j) {
            all[t].score = (double)scores[(int64_t)h * T + j];
            all[t].cell = h;
            all[t].pos = j;
            ++t;
        }
    qsort(all, (size_t)nc, sizeof(cand), cmp_cand);
    int64_t K = total_budget - nfloor;
    unsigned char *kept = (unsigned char *)calloc((size_t)cells * T, 1);
    for (int h = 0; h < cells; ++h)
        for (int j = T - F; j < T; ++j)
            kept[(int64_t)h * T + j] = 1;
    for (int64_t q = 0; q < K; ++q)
        kept[(int64_t)all[q].cell * T + all[q].pos] = 1;
    if (tau)
        *tau = K > 0 ? (float)all[K - 1].score : INFINITY;
    int64_t acc = 0;
    for (int h = 0; h < cells; ++h) {
        int cnt = 0;
        if (offsets)
            offsets[h] = acc;
        for (int j = 0; j < T; ++j)
            if (kept[(int64_t)h * T + j]) {
                if (kept_pos)
                    kept_pos[acc + cnt] = j;
                ++cnt;
            }
        if (counts)
            counts[h] = cnt;
        acc += cnt;
    }
    if (offsets)
        offsets[cells] = acc;
    /* per-cell dropped mass of the normalised scores */
    keyed *o = (keyed *)malloc(sizeof(keyed) * (size_t)T);
    for (int h = 0; h < cells; ++h) {
        const float *s = scores + (int64_t)h * T;
        double tot = 0.0, da = 0.0, du = 0.0;
        for (int j = 0; j < T; ++j)
            tot += (double)s[j];
        for (int j = 0; j < T; ++j)
            if (!kept[(int64_t)h * T + j])
                da += (double)s[j];
        for (int j = 0; j < T; ++j) {
            o[j].key = (double)s[j];
            o[j].idx = j;
        }
        qsort(o, (size_t)T, sizeof(keyed), cmp_desc_key_asc_idx);
        int su = uniform_s < T ? uniform_s : T;
        for (int q = su; q < T; ++q)
            du += o[q].key;
        if (dropped_alloc)
            dropped_alloc[h] = tot > 0 ? da / tot : 0.0;
        if (dropped_uniform)
            dropped_uniform[h] = tot > 0 ? du / tot : 0.0;
    }
    free(o);
    free(kept);
    free(all);
    return ORC_OK;
}

/* f3: ContourKV with its budget enforced per cell (Sec. 4: enforcement caps
 * every head at a uniform method's per-head count).  Step 1 is the plain
 * allocation above (orc_contour_alloc, which also gives tau and the
 * uniform-budget dropped mass); step 2 truncates each cell: its floor stays,
 * and of its kept non-floor positions only the best cap - |F| under
 * (score desc, position asc) remain.  Outputs as orc_contour_alloc, with
 * counts[h] = min(allocated count, cap), offsets over those counts and
 * dropped_alloc the mass outside the truncated set.  kept_pos needs room for
 * total_budget entries.  Requires cap >= |F|. */
int orc_contour_alloc_capped(const float *scores, int cells, int T, int floor_, int64_t total_budget,
                             int uniform_s, int cap, int32_t *counts, int64_t *offsets, int32_t *kept_pos,
                             float *tau, double *dropped_uniform, double *dropped_alloc)
{
    const int F = floor_ < T ? floor_ : T;
    if (cap < F)
        return ORC_ERR_ARG;
    int32_t *c0 = (int32_t *)malloc(sizeof(int32_t) * (size_t)cells);
    int64_t *o0 = (int64_t *)malloc(sizeof(int64_t) * ((size_t)cells + 1));
    int32_t *p0 = (int32_t *)malloc(sizeof(int32_t) * (size_t)(total_budget > 0 ? total_budget : 1));
    int st = orc_contour_alloc(scores, cells, T, floor_, total_budget, uniform_s, c0, o0, p0, tau,
                               dropped_uniform, NULL);
    if (st) {
        free(c0);
        free(o0);
        free(p0);
        return st;
    }
    keyed *nf = (keyed *)malloc(sizeof(keyed) * (size_t)T);
    unsigned char *kept = (unsigned char *)malloc((size_t)T);
    int64_t acc = 0;
    for (int h = 0; h < cells; ++h) {
        const float *s = scores + (int64_t)h * T;
        memset(kept, 0, (size_t)T);
        int m = 0;
        for (int64_t q = o0[h]; q < o0[h + 1]; ++q) {
            const int j = p0[q];
            if (j >= T - F) {
                kept[j] = 1; /* the floor */
            } else {
                nf[m].key = (double)s[j];
                nf[m].idx = j;
                ++m;
            }
        }
        qsort(nf, (size_t)m, sizeof(keyed), cmp_desc_key_asc_idx);
        const int keep = m < cap - F ? m : cap - F;
        for (int t = 0; t < keep; ++t)
            kept[nf[t].idx] = 1;
        int cnt = 0;
        double tot = 0.0, da = 0.0;
        offsets[h] = acc;
        for (int j = 0; j < T; ++j) {
            tot += (double)s[j];
            if (kept[j])
                kept_pos[acc + cnt++] = j;
            else
                da += (double)s[j];
        }
        counts[h] = cnt;
        acc += cnt;
        if (dropped_alloc)
            dropped_alloc[h] = tot > 0 ? da / tot : 0.0;
    }
    offsets[cells] = acc;
    free(kept);
    free(nf);
    free(c0);
    free(o0);
    free(p0);
    return ORC_OK;
}

/* a8: ragged per-head storage (Sec. 4): the kept rows of every cell, copied
 * byte for byte, cells in order, positions ascending.  K, V: [cells][T][d]
 * of elem_bytes each; outputs [offsets[cells]][d]. */
int orc_ragged_compact(const void *K, const void *V, int cells, int T, int d, int elem_bytes,
                       const int64_t *offsets, const int32_t *kept_pos, void *K_out, void *V_out)
{
    size_t row = (size_t)d * (size_t)elem_bytes;
    for (int h = 0; h < cells; ++h)
        for (int64_t q = offsets[h]; q < offsets[h + 1]; ++q) {
            int j = kept_pos[q];
            if (j < 0 || j >= T)
                return ORC_ERR_ARG;
            size_t src = ((size_t)h * (size_t)T + (size_t)j) * row;
            memcpy((char *)K_out + (size_t)q * row, (const char *)K + src, row);
            memcpy((char *)V_out + (size_t)q * row, (const char *)V + src, row);
        }
    return ORC_OK;
}

/* ------------------------------------------------- candidate-set search */

/* The candidate set of Definition 2.2 for budget k: the top-mass set plus the
 * E dropped keys of largest single-key error p_j ||v_j - mu|| (ties -> lower
 * index).  pool receives the members in ascending key order; returns their
 * number.  *margin = (e_E - e_{E+1}) / e_E at the pool boundary (+inf when
 * every dropped key joins the pool or E = 0). */
static int candidate_set(const instance *I, int k, int E, unsigned char *in_A, int *pool, double *margin)
{
    const int n = I->n, d = I->d;
    topk_by_logit(n, I->logit, k, in_A);
    keyed *err = (keyed *)malloc(sizeof(keyed) * ((size_t)n + 1));
    int nd = 0;
    for (int j = 0; j < n; ++j) {
        if (in_A[j])
            continue;
        double s2 = 0.0;
        for (int c = 0; c < d; ++c) {
            double t = I->v[(int64_t)j * d + c] - I->mu[c];
            s2 += t * t;
        }
        err[nd].key = I->p[j] * sqrt(s2);
        err[nd].idx = j;
        ++nd;
    }
    qsort(err, (size_t)nd, sizeof(keyed), cmp_desc_key_asc_idx);
    *margin = (E > 0 && E < nd) ? (err[E - 1].key > 0 ? (err[E - 1].key - err[E].key) / err[E - 1].key : 0.0)
                                : INFINITY;
    unsigned char *in_pool = (unsigned char *)malloc((size_t)n + 1);
    memcpy(in_pool, in_A, (size_t)n);
    for (int t = 0; t < E && t < nd; ++t)
        in_pool[err[t].idx] = 1;
    int P = 0;
    for (int j = 0; j < n; ++j)
        if (in_pool[j])
            pool[P++] = j;
    free(in_pool);
    free(err);
    return P;
}

/* f2: ES_pool(k) (Definition 2.2), the exact minimum of es over the size-k
 * subsets of the candidate set, by exhaustive enumeration in lexicographic
 * order with es of every subset from its definition (m_A = N_A / p(A) with the
 * row's own masses and mu).  Exact ties -> the smallest colex rank of the
 * members' positions in the candidate set (sorted by key index).
 * k: [rows][nb]; E: [nb] extras of budget slot b.
 * Outputs: best_gap [rows][nb] = ES_pool; best_idx [rows][nb][k_max]
 * ascending key indices (-1 past k); topk_gap [rows][nb] = es(A*_k);
 * second_gap [rows][nb] the second-smallest es over the enumerated subsets
 * (+inf if there is one subset); n_subsets [rows][nb] = C(|pool|, k);
 * pool_margin [rows][nb] the relative gap between the E-th and the (E+1)-th
 * single-key error of the dropped keys (+inf if all join); status [rows].  Returns ORC_ERR_ARG for a budget out of range, k > k_max, or more
 * than max_subsets subsets in a pool. */
int orc_pool_best_subset(const orc_rows *R, int nb, const int32_t *k, const int32_t *E, int k_max,
                         int64_t max_subsets, double *best_gap, int32_t *best_idx, double *topk_gap,
                         double *second_gap, int64_t *n_subsets, double *pool_margin, int32_t *status)
{
    int64_t rows = R->num_groups * R->rows_per_group;
    int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad)
    for (int64_t r = 0; r < rows; ++r) {
        instance I;
        int st = load_row(R, r, &I);
        status[r] = st;
        if (st) {
            instance_free(&I);
            continue;
        }
        const int n = I.n;
        unsigned char *in_A = (unsigned char *)malloc((size_t)n + 1);
        int *pool = (int *)malloc(sizeof(int) * ((size_t)n + 1));
        int *c = (int *)malloc(sizeof(int) * ((size_t)n + 1));
        int *mem = (int *)malloc(sizeof(int) * ((size_t)n + 1));
        double *NA = (double *)malloc(sizeof(double) * (size_t)I.d);
        for (int b = 0; b < nb; ++b) {
            const int64_t rb = r * nb + b;
            const int kb = k[rb];
            if (kb < 1 || kb > n || kb > k_max || E[b] < 0) {
                bad |= 1;
                continue;
            }
            double pm;
            const int P = candidate_set(&I, kb, E[b], in_A, pool, &pm);
            if (pool_margin)
                pool_margin[rb] = pm;
            const uint64_t cnt = binom(P, kb);
            if (n_subsets)
                n_subsets[rb] = (int64_t)cnt;
            if (cnt > (uint64_t)max_subsets) {
                bad |= 1;
                continue;
            }
            if (topk_gap)
                topk_gap[rb] = eval_set(&I, in_A, NULL).gap;
            double best = INFINITY, second = INFINITY;
            uint64_t best_rank = 0;
            int32_t *bi = best_idx + rb * (int64_t)k_max;
            for (int t = 0; t < kb; ++t)
                c[t] = t;
            for (;;) {
                for (int t = 0; t < kb; ++t)
                    mem[t] = pool[c[t]];
                const double es = es_of_members(&I, mem, kb, NA);
                uint64_t rank = 0;
                for (int t = 0; t < kb; ++t)
                    rank += binom(c[t], t + 1);
                if (es < best || (es == best && rank < best_rank)) {
                    second = best < second ? best : second;
                    best = es;
                    best_rank = rank;
                    for (int t = 0; t < kb; ++t)
                        bi[t] = mem[t];
                } else if (es < second) {
                    second = es;
                }
                /* next combination in lexicographic order */
                int t = kb - 1;
                while (t >= 0 && c[t] == P - kb + t)
                    --t;
                if (t < 0)
                    break;
                ++c[t];
                for (int u = t + 1; u < kb; ++u)
                    c[u] = c[u - 1] + 1;
            }
            for (int t = kb; t < k_max; ++t)
                bi[t] = -1;
            best_gap[rb] = best;
            if (second_gap)
                second_gap[rb] = second;
        }
        free(NA);
        free(mem);
        free(c);
        free(pool);
        free(in_A);
        instance_free(&I);
    }
    return bad ? ORC_ERR_ARG : ORC_OK;
}

/* The candidate set of Definition 2.2 for row r at budget k (the helper
 * above, exposed for the tests): pool (capacity n of the row) receives the
 * members in ascending key order, the return value is their number (negative
 * on a bad row or budget), *margin the pool-boundary margin. */
int orc_candidate_set(const orc_rows *R, int64_t r, int k, int E, int32_t *pool, double *margin)
{
    instance I;
    if (load_row(R, r, &I)) {
        instance_free(&I);
        return -1;
    }
    if (k < 1 || k > I.n || E < 0) {
        instance_free(&I);
        return -1;
    }
    unsigned char *in_A = (unsigned char *)malloc((size_t)I.n + 1);
    int *pl = (int *)malloc(sizeof(int) * ((size_t)I.n + 1));
    const int P = candidate_set(&I, k, E, in_A, pl, margin);
    for (int t = 0; t < P; ++t)
        pool[t] = pl[t];
    free(pl);
    free(in_A);
    instance_free(&I);
    return P;
}

/* One round of the balancing selector (Sec. 2.1), every option scored: for
 * row r and the kept set in_A (n bytes of the row), es(A - i + j) for every
 * kept key i (ascending) and every j in add[0..nadd), from the definition
 * m_A' = N_A' / p(A') with N_A' = N_A - p_i v_i + p_j v_j.  Writes
 * es_out[a * nadd + q] for the a-th kept key and add[q], and *cur = es(A).
 * Keys of add that are already in A are scored as given (the tests pass keys
 * outside A).  Returns the number of kept keys, or -1 on a bad row. */
int orc_swap_scores(const orc_rows *R, int64_t r, const unsigned char *in_A, const int32_t *add, int nadd,
                    double *es_out, double *cur)
{
    instance I;
    if (load_row(R, r, &I)) {
        instance_free(&I);
        return -1;
    }
    const int n = I.n, d = I.d;
    double *NA = (double *)calloc((size_t)d, sizeof(double));
    int *kept = (int *)malloc(sizeof(int) * ((size_t)n + 1));
    double PA = 0.0;
    int na = 0;
    for (int j = 0; j < n; ++j)
        if (in_A[j]) {
            kept[na++] = j;
            PA += I.p[j];
            for (int c = 0; c < d; ++c)
                NA[c] += I.p[j] * I.v[(int64_t)j * d + c];
        }
    if (cur) {
        double g2 = 0.0;
        for (int c = 0; c < d; ++c) {
            const double diff = NA[c] / PA - I.mu[c];
            g2 += diff * diff;
        }
        *cur = sqrt(g2);
    }
#pragma omp parallel for schedule(static)
    for (int a = 0; a < na; ++a) {
        const int i = kept[a];
        for (int q = 0; q < nadd; ++q) {
            const int j = add[q];
            const double P2 = PA - I.p[i] + I.p[j];
            double g2 = 0.0;
            for (int c = 0; c < d; ++c) {
                const double Nc = NA[c] - I.p[i] * I.v[(int64_t)i * d + c] + I.p[j] * I.v[(int64_t)j * d + c];
                const double diff = Nc / P2 - I.mu[c];
                g2 += diff * diff;
            }
            es_out[(int64_t)a * nadd + q] = sqrt(g2);
        }
    }
    free(kept);
    free(NA);
    instance_free(&I);
    return na;
}

/* f3: ragged storage with room per cell (Sec. 4, ragged storage; Sec. 1,
 * the multi-turn cache that decode keeps appending to).  Cell h owns rows
 * base[h] .. base[h] + capacity[h] - 1 of the store.
 * orc_ragged_compact_to: cell h's kept rows (offsets[h] .. offsets[h+1] - 1
 * of kept_pos) copied byte for byte to its rows from base[h] on, when they
 * fit (status[h] = 0), else nothing copied and status[h] = 1.
 * orc_ragged_append: m new rows per cell ([cells][m] rows of row_bytes)
 * copied behind the counts[h] filled rows, counts[h] += m, when they fit
 * (status[h] = 0), else nothing and status[h] = 1. */
int orc_ragged_compact_to(const void *K, const void *V, int cells, int T, int row_bytes, const int64_t *offsets,
                          const int32_t *kept_pos, const int64_t *base, const int32_t *capacity, void *K_store,
                          void *V_store, int32_t *status)
{
    for (int h = 0; h < cells; ++h) {
        const int64_t cnt = offsets[h + 1] - offsets[h];
        status[h] = cnt <= capacity[h] ? 0 : 1;
        if (status[h])
            continue;
        for (int64_t q = 0; q < cnt; ++q) {
            const int j = kept_pos[offsets[h] + q];
            if (j < 0 || j >= T)
                return ORC_ERR_ARG;
            const size_t src = ((size_t)h * T + (size_t)j) * (size_t)row_bytes;
            const size_t dst = (size_t)(base[h] + q) * (size_t)row_bytes;
            memcpy((char *)K_store + dst, (const char *)K + src, (size_t)row_bytes);
            memcpy((char *)V_store + dst, (const char *)V + src, (size_t)row_bytes);
        }
    }
    return ORC_OK;
}

int orc_ragged_append(void *K_store, void *V_store, const int64_t *base, const int32_t *capacity, int32_t *counts,
                      const void *new_K, const void *new_V, int cells, int m, int row_bytes, int32_t *status)
{
    for (int h = 0; h < cells; ++h) {
        status[h] = (counts[h] >= 0 && (int64_t)counts[h] + m <= (int64_t)capacity[h]) ? 0 : 1;
        if (status[h])
            continue;
        for (int t = 0; t < m; ++t) {
            const size_t src = ((size_t)h * m + (size_t)t) * (size_t)row_bytes;
            const size_t dst = (size_t)(base[h] + counts[h] + t) * (size_t)row_bytes;
            memcpy((char *)K_store + dst, (const char *)new_K + src, (size_t)row_bytes);
            memcpy((char *)V_store + dst, (const char *)new_V + src, (size_t)row_bytes);
        }
        counts[h] += m;
    }
    return ORC_OK;
}

/* f3: the observation-window importance score (Sec. 4 runs ContourKV with
 * SnapKV's window score).  Per cell c: window queries q_i (i < w, bf16 bits,
 * query i at position T - w + i seeing keys j <= T - w + i) and keys k_j
 * (bf16 bits); a_ij = softmax over the visible j of scale * q_i . k_j (fp64),
 * vote_j = sum_i a_ij; scores_j = max of vote over [j - pool/2, j + pool/2]
 * clipped to the prefix [0, T - w) for prefix positions, vote_j in the
 * window.  votes may be NULL. */
static double bf16_at(const uint16_t *p, size_t i)
{
    uint32_t bits = ((uint32_t)p[i]) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

int orc_window_score(const uint16_t *Qw, const uint16_t *K, int cells, int T, int d, int w, double scale, int pool,
                     double *scores, double *votes)
{
    if (cells < 1 || T < 1 || d < 1 || w < 1 || w > T || pool < 1 || pool % 2 == 0)
        return ORC_ERR_ARG;
#pragma omp parallel for schedule(dynamic, 1)
    for (int c = 0; c < cells; ++c) {
        double *vote = (double *)calloc((size_t)T, sizeof(double));
        double *L = (double *)malloc(sizeof(double) * (size_t)T);
        for (int i = 0; i < w; ++i) {
            const int last = T - w + i; /* the query's own position */
            double M = -INFINITY, Z = 0.0;
            for (int j = 0; j <= last; ++j) {
                double dot = 0.0;
                for (int e = 0; e < d; ++e)
                    dot += bf16_at(Qw, ((size_t)c * w + i) * d + e) * bf16_at(K, ((size_t)c * T + j) * d + e);
                L[j] = scale * dot;
                if (L[j] > M)
                    M = L[j];
            }
            for (int j = 0; j <= last; ++j)
                Z += exp(L[j] - M);
            for (int j = 0; j <= last; ++j)
                vote[j] += exp(L[j] - M) / Z;
        }
        const int lim = T - w, h = pool / 2;
        for (int j = 0; j < T; ++j) {
            double r = vote[j];
            if (j < lim)
                for (int q = j - h; q <= j + h; ++q)
                    if (q >= 0 && q < lim && vote[q] > r)
                        r = vote[q];
            scores[(size_t)c * T + j] = r;
            if (votes)
                votes[(size_t)c * T + j] = vote[j];
        }
        free(L);
        free(vote);
    }
    return ORC_OK;
}

/* f4: the deployed selectors audited in Sec. 2.3 with App. C's settings, each
 * a kept set scored with es (Definition 2.1).  For budget s:
 *   StreamingLLM: positions j < min(4, s/2) and j >= n - (s - min(4, s/2));
 *   H2O: positions j >= n - s/2, and of j < n - s/2 the s - s/2 of largest
 *        accumulated mass G_j = sum over the group's rows of p_ij;
 *   SnapKV: w = max(1, min(32, s/2)); positions j >= n - w, and of j < n - w
 *        the s - w of largest pooled vote max_{|q - j| <= 3, q < n - w} vote_q,
 *        vote_q = sum over the group's last min(w, R) rows of p_iq;
 *   Quest (P = max(2, s/4)) and Quest-16 (P = 16, s >= 16): the floor(s/P)
 *        pages of P consecutive keys with the largest maximum logit.
 * Equal scores: lower position (page) first.  es NaN when the set is empty.
 * Outputs: es [rows][5][nb]; bits [rows][5][nb][words] (may be NULL); G
 * [groups][max_n] and pooled [groups][nb][max_n] (may be NULL; pooled is the
 * vote itself at the window positions). */
/* mark the first `take` entries of a sorted candidate list */
static void mark_first(const keyed *a, int m, int take, unsigned char *in)
{
    for (int t = 0; t < take && t < m; ++t)
        in[a[t].idx] = 1;
}

int orc_selector_audit(const orc_rows *R, int nb, const int32_t *s, int max_n, double *es, uint32_t *bits, int words,
                       double *G_out, double *pooled_out)
{
    const int64_t groups = R->num_groups;
    const int Rg = R->rows_per_group;
    int bad = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(| : bad)
    for (int64_t g = 0; g < groups; ++g) {
        const int n = R->n[g];
        double *G = (double *)calloc((size_t)n + 1, sizeof(double));
        double *vote = (double *)calloc((size_t)nb * n + 1, sizeof(double));
        double *pooled = (double *)calloc((size_t)nb * n + 1, sizeof(double));
        unsigned char *hset = (unsigned char *)calloc((size_t)nb * n + 1, 1);
        unsigned char *sset = (unsigned char *)calloc((size_t)nb * n + 1, 1);
        unsigned char *in = (unsigned char *)calloc((size_t)n + 1, 1);
        keyed *o = (keyed *)malloc(sizeof(keyed) * ((size_t)n + 1));
        /* accumulated masses and window votes over the group's rows */
        for (int i = 0; i < Rg; ++i) {
            instance I;
            if (load_row(R, g * Rg + i, &I)) {
                instance_free(&I);
                bad |= 1;
                continue;
            }
            for (int j = 0; j < n; ++j) {
                G[j] += I.p[j];
                for (int b = 0; b < nb; ++b) {
                    int w = s[b] / 2 < 32 ? s[b] / 2 : 32;
                    w = w < 1 ? 1 : w;
                    if (i >= Rg - w)
                        vote[(size_t)b * n + j] += I.p[j];
                }
            }
            instance_free(&I);
        }
        /* the group-level sets */
        for (int b = 0; b < nb; ++b) {
            const int sb = s[b];
            if (sb < 1 || sb > n)
                continue;
            const int r = sb / 2;
            for (int j = 0; j < n - r; ++j) {
                o[j].key = G[j];
                o[j].idx = j;
            }
            qsort(o, (size_t)(n - r), sizeof(keyed), cmp_desc_key_asc_idx);
            mark_first(o, n - r, sb - r, hset + (size_t)b * n);
            for (int j = n - r; j < n; ++j)
                hset[(size_t)b * n + j] = 1;
            int w = sb / 2 < 32 ? sb / 2 : 32;
            w = w < 1 ? 1 : w;
            const int lim = n - w;
            for (int j = 0; j < n; ++j) {
                double v = vote[(size_t)b * n + j];
                if (j < lim)
                    for (int q = j - 3; q <= j + 3; ++q)
                        if (q >= 0 && q < lim && vote[(size_t)b * n + q] > v)
                            v = vote[(size_t)b * n + q];
                pooled[(size_t)b * n + j] = v;
            }
            for (int j = 0; j < lim; ++j) {
                o[j].key = pooled[(size_t)b * n + j];
                o[j].idx = j;
            }
            qsort(o, (size_t)lim, sizeof(keyed), cmp_desc_key_asc_idx);
            mark_first(o, lim, sb - w, sset + (size_t)b * n);
            for (int j = lim; j < n; ++j)
                sset[(size_t)b * n + j] = 1;
        }
        if (G_out)
            for (int j = 0; j < n; ++j)
                G_out[g * max_n + j] = G[j];
        if (pooled_out)
            for (int b = 0; b < nb; ++b)
                for (int j = 0; j < n; ++j)
                    pooled_out[(g * nb + b) * max_n + j] = pooled[(size_t)b * n + j];
        /* every row: the five sets and their es */
        for (int i = 0; i < Rg; ++i) {
            const int64_t row = g * Rg + i;
            instance I;
            if (load_row(R, row, &I)) {
                instance_free(&I);
                continue;
            }
            for (int b = 0; b < nb; ++b) {
                const int sb = s[b];
                for (int sel = 0; sel < 5; ++sel) {
                    memset(in, 0, (size_t)n);
                    int any = sb >= 1 && sb <= n;
                    if (any && sel == 0) {
                        const int sinks = sb / 2 < 4 ? sb / 2 : 4;
                        for (int j = 0; j < n; ++j)
                            in[j] = j < sinks || j >= n - (sb - sinks);
                    } else if (any && sel == 1) {
                        memcpy(in, hset + (size_t)b * n, (size_t)n);
                    } else if (any && sel == 2) {
                        memcpy(in, sset + (size_t)b * n, (size_t)n);
                    } else if (any) {
                        const int P = sel == 3 ? (sb / 4 > 2 ? sb / 4 : 2) : 16;
                        const int np = (n + P - 1) / P, mp = sb / P;
                        if (sel == 4 && sb < 16)
                            any = 0;
                        if (mp < 1)
                            any = 0;
                        if (any) {
                            for (int p = 0; p < np; ++p) {
                                double m = -INFINITY;
                                for (int j = p * P; j < n && j < p * P + P; ++j)
                                    if ((double)I.logit[j] > m)
                                        m = (double)I.logit[j];
                                o[p].key = m;
                                o[p].idx = p;
                            }
                            qsort(o, (size_t)np, sizeof(keyed), cmp_desc_key_asc_idx);
                            for (int t = 0; t < mp && t < np; ++t)
                                for (int j = o[t].idx * P; j < n && j < o[t].idx * P + P; ++j)
                                    in[j] = 1;
                        }
                    }
                    int cnt = 0;
                    for (int j = 0; j < n; ++j)
                        cnt += in[j];
                    es[(row * 5 + sel) * nb + b] = cnt > 0 ? eval_set(&I, in, NULL).gap : NAN;
                    if (bits) {
                        uint32_t *wv = bits + ((row * 5 + sel) * nb + b) * (int64_t)words;
                        for (int t = 0; t < words; ++t)
                            wv[t] = 0u;
                        for (int j = 0; j < n; ++j)
                            if (in[j])
                                wv[j >> 5] |= 1u << (j & 31);
                    }
                }
            }
            instance_free(&I);
        }
        free(o);
        free(in);
        free(sset);
        free(hset);
        free(pooled);
        free(vote);
        free(G);
    }
    return bad ? ORC_ERR_ARG : ORC_OK;
}

/* ---------------------------------------------------------- group vote */

/* f1: the group vote (Sec. 2.1, shared kept sets).  Deployment keeps one set
 * per KV head for all the query rows that share it; the vote keeps the s keys
 * of largest mass summed over the group's rows,
 *     G_j = sum_{rows i of the group} p_ij,
 * equal G -> lower index first (the same tie reading as the top-mass set).
 * Every row of the group is then scored against that one set with the
 * Definition 2.1 / Sec. 2.1 quantities (es and dropped mass of the row's own
 * masses).  With one row per group the vote is the row's own top-mass set.
 * s: [groups][nb], 1 <= s <= n[g].
 * Outputs (any may be NULL except status):
 *   mass [groups][max_n]      G (entries past n[g] untouched),
 *   margin [groups][nb]       (G_(s) - G_(s+1)) / G_(s) of the order, the
 *                             relative gap between the last kept and the first
 *                             dropped key (1 when s = n, 0 when G_(s) = 0),
 *   bits [groups][nb][words]  bit j%32 of word j/32 = (j in the vote set),
 *   gap, dropped [rows][nb]   es(A) and sum_{j not in A} p_j of each row,
 *   status [rows]             0, ORC_ERR_ARG (a budget of its group is out of
 *                             range) or ORC_ERR_NONFINITE (a logit of its group
 *                             is not finite).
 * eval: [rows] or NULL; rows with eval[r] == 0 skip the per-row scoring (the
 * group's G and set still use every row). */
int orc_group_vote(const orc_rows *R, int nb, const int32_t *s, int max_n, const unsigned char *eval,
                   double *mass, double *margin, uint32_t *bits, int words, double *gap,
                   double *dropped, int32_t *status)
{
    const int64_t G = R->num_groups, RPG = R->rows_per_group;
    unsigned char *sets = (unsigned char *)calloc((size_t)(G * nb * (int64_t)max_n) + 1, 1);
    int32_t *gst = (int32_t *)calloc((size_t)G + 1, sizeof(int32_t));
    /* the vote set of every group and budget */
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t g = 0; g < G; ++g) {
        const int n = R->n[g];
        double *Gm = (double *)calloc((size_t)n + 1, sizeof(double));
        double *p = (double *)malloc(sizeof(double) * ((size_t)n + 1));
        for (int64_t i = 0; i < RPG && !gst[g]; ++i) {
            const float *l = R->logits + R->logit_off[g] + i * (int64_t)n;
            if (softmax_f64(n, l, p))
                gst[g] = ORC_ERR_NONFINITE;
            else
                for (int j = 0; j < n; ++j)
                    Gm[j] += p[j];
        }
        if (mass)
            for (int j = 0; j < n; ++j)
                mass[g * (int64_t)max_n + j] = Gm[j];
        keyed *o = (keyed *)malloc(sizeof(keyed) * ((size_t)n + 1));
        for (int j = 0; j < n; ++j) {
            o[j].key = Gm[j];
            o[j].idx = j;
        }
        qsort(o, (size_t)n, sizeof(keyed), cmp_desc_key_asc_idx);
        for (int b = 0; b < nb; ++b) {
            const int sb = s[g * nb + b];
            const int64_t gb = g * nb + b;
            if (sb < 1 || sb > n) {
                if (!gst[g])
                    gst[g] = ORC_ERR_ARG;
                continue;
            }
            unsigned char *in_A = sets + gb * (int64_t)max_n;
            for (int t = 0; t < sb; ++t)
                in_A[o[t].idx] = 1;
            if (margin) {
                const double last = o[sb - 1].key;
                margin[gb] = sb == n ? 1.0 : (last > 0 ? (last - o[sb].key) / last : 0.0);
            }
            if (bits) {
                uint32_t *w = bits + gb * (int64_t)words;
                for (int t = 0; t < words; ++t)
                    w[t] = 0u;
                for (int j = 0; j < n; ++j)
                    if (in_A[j])
                        w[j >> 5] |= 1u << (j & 31);
            }
        }
        free(o);
        free(p);
        free(Gm);
    }
    /* every row against its group's sets */
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t r = 0; r < G * RPG; ++r) {
        const int64_t g = r / RPG;
        status[r] = gst[g];
        if (gst[g] || (eval && !eval[r]))
            continue;
        instance I;
        int st = load_row(R, r, &I);
        if (st) {
            status[r] = st;
            instance_free(&I);
            continue;
        }
        for (int b = 0; b < nb; ++b) {
            set_eval e = eval_set(&I, sets + (g * nb + b) * (int64_t)max_n, NULL);
            if (gap) gap[r * nb + b] = e.gap;
            if (dropped) dropped[r * nb + b] = e.dropped;
        }
        instance_free(&I);
    }
    free(gst);
    free(sets);
    return ORC_OK;
}

#ifdef _OPENMP
#include <omp.h>
#endif

/* threads the OpenMP loops above use */
int orc_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
