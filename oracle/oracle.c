/*
 * oracle.c -- plain, slow, fp64 reference for ragged causal grouped-query
 * prefill attention.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing in the product path may call, link or
 * load this file; only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg use it.  It shares no code, header or constant with the
 * CUDA library.
 *
 * What it computes (OpScale, §2.1 "Compute Sensitivity" and "Memory
 * Sensitivity"): the attention operator is exact softmax attention, O(L^2 b)
 * in the prompt length L; FlashAttention only avoids materialising the L x L
 * score matrix, it does not change the result.  This file therefore writes
 * the plain definition out, one output row at a time, with the whole row of
 * scores materialised and an explicit two-pass softmax:
 *
 *   sequence s, query row i in [0, Lq_s), query head h, kv head g = h / G,
 *   G = Hq / Hkv (contiguous head groups; §5.6 names the switch from
 *   multi-head to grouped-query attention),
 *   delta_s = Lk_s - Lq_s (bottom-right alignment, so that a chunk of a
 *   prompt attends to its prefix: chunked prefill, §6),
 *   visible keys J = { j : 0 <= j <= i + delta_s and j < Lk_s },
 *   x_j   = scale * sum_c q[i,h,c] * k[j,g,c]
 *   m     = max_j x_j,  p_j = exp(x_j - m),  l = sum_j p_j
 *   O[i,h,:] = sum_j p_j v[j,g,:] / l,   LSE[i,h] = m + ln(l)
 *   J empty  ->  O = 0, LSE = -infinity.
 *
 * Inputs are bf16 bit patterns (uint16); every value is widened exactly to
 * double.  Layouts: q [total_q, Hq, d], k and v [total_k, Hkv, d], all
 * packed; cu_q / cu_k hold n_seq + 1 prefix offsets.
 *
 * Parity pins (test suite, CPU): length-1 rows, constant V, zero queries,
 * a hand-derived worked example, a dense masked-matrix formulation through
 * scipy on tiny inputs, chunk consistency, head-mapping and sequence
 * permutation invariants, and rows that see no key.  A mutation test plants
 * plausible mistakes in copies of this file and checks that a pin fails for
 * each.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

static double widen_bf16(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Index of the sequence that owns packed query token `token`, or -1. */
static int32_t owner_sequence(const int32_t *cu_q, int32_t n_seq, int64_t token)
{
    for (int32_t s = 0; s < n_seq; ++s)
        if (token >= cu_q[s] && token < cu_q[s + 1])
            return s;
    return -1;
}

/*
 * One output row.  `x` is caller scratch of at least Lk_s doubles (the
 * materialised score row).  Returns 0 on success, -1 if the token is outside
 * every sequence.
 */
int oracle_row(const uint16_t *q, const uint16_t *k, const uint16_t *v,
               const int32_t *cu_q, const int32_t *cu_k, int32_t n_seq,
               int32_t Hq, int32_t Hkv, int32_t d, double scale,
               int64_t token, int32_t h, double *o_row, double *lse, double *x)
{
    int32_t s = owner_sequence(cu_q, n_seq, token);
    if (s < 0 || h < 0 || h >= Hq)
        return -1;
    int64_t Lq = cu_q[s + 1] - cu_q[s];
    int64_t Lk = cu_k[s + 1] - cu_k[s];
    int64_t delta = Lk - Lq;
    int64_t i = token - cu_q[s];
    int32_t G = Hq / Hkv;
    int32_t g = h / G;

    /* visible keys: 0 <= j <= i + delta and j < Lk */
    int64_t last = i + delta;
    if (last > Lk - 1)
        last = Lk - 1;
    int64_t n_vis = last + 1; /* may be <= 0 */

    const uint16_t *qrow = q + (token * Hq + h) * (int64_t)d;

    if (n_vis <= 0) {
        for (int32_t c = 0; c < d; ++c)
            o_row[c] = 0.0;
        *lse = -INFINITY;
        return 0;
    }

    /* pass 1: scores and their maximum */
    double m = -INFINITY;
    for (int64_t j = 0; j < n_vis; ++j) {
        const uint16_t *krow = k + ((cu_k[s] + j) * Hkv + g) * (int64_t)d;
        double dot = 0.0;
        for (int32_t c = 0; c < d; ++c)
            dot += widen_bf16(qrow[c]) * widen_bf16(krow[c]);
        x[j] = scale * dot;
        if (x[j] > m)
            m = x[j];
    }

    /* pass 2: exponentials, their sum, and the weighted sum of value rows */
    double l = 0.0;
    for (int32_t c = 0; c < d; ++c)
        o_row[c] = 0.0;
    for (int64_t j = 0; j < n_vis; ++j) {
        double p = exp(x[j] - m);
        l += p;
        const uint16_t *vrow = v + ((cu_k[s] + j) * Hkv + g) * (int64_t)d;
        for (int32_t c = 0; c < d; ++c)
            o_row[c] += p * widen_bf16(vrow[c]);
    }
    for (int32_t c = 0; c < d; ++c)
        o_row[c] /= l;
    *lse = m + log(l);
    return 0;
}

/* ---- row-parallel driver (harness only: threads split the row list) ---- */

struct row_job {
    const uint16_t *q, *k, *v;
    const int32_t *cu_q, *cu_k;
    int32_t n_seq, Hq, Hkv, d;
    double scale;
    const int64_t *tokens;
    const int32_t *heads;
    int64_t n_rows;
    double *o, *lse;
    int64_t max_lk;
    int64_t next; /* shared row counter */
    pthread_mutex_t lock;
    int failed;
};

static void *row_worker(void *arg)
{
    struct row_job *job = (struct row_job *)arg;
    double *x = (double *)malloc(sizeof(double) * (size_t)(job->max_lk > 0 ? job->max_lk : 1));
    if (!x) {
        job->failed = 1;
        return NULL;
    }
    for (;;) {
        int64_t r0;
        pthread_mutex_lock(&job->lock);
        r0 = job->next;
        job->next += 16;
        pthread_mutex_unlock(&job->lock);
        if (r0 >= job->n_rows)
            break;
        int64_t r1 = r0 + 16 < job->n_rows ? r0 + 16 : job->n_rows;
        for (int64_t r = r0; r < r1; ++r) {
            if (oracle_row(job->q, job->k, job->v, job->cu_q, job->cu_k, job->n_seq,
                           job->Hq, job->Hkv, job->d, job->scale, job->tokens[r],
                           job->heads[r], job->o + r * job->d, job->lse + r, x) != 0)
                job->failed = 1;
        }
    }
    free(x);
    return NULL;
}

/*
 * Selected rows: row r is (tokens[r], heads[r]); o receives n_rows x d
 * doubles and lse n_rows doubles.  Returns 0, or -1 on a bad argument.
 */
int oracle_attention_rows(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                          const int32_t *cu_q, const int32_t *cu_k, int32_t n_seq,
                          int32_t Hq, int32_t Hkv, int32_t d, double scale,
                          const int64_t *tokens, const int32_t *heads, int64_t n_rows,
                          double *o, double *lse, int32_t n_threads)
{
    if (n_seq < 0 || Hq <= 0 || Hkv <= 0 || Hq % Hkv != 0 || d <= 0)
        return -1;
    struct row_job job;
    memset(&job, 0, sizeof job);
    job.q = q; job.k = k; job.v = v;
    job.cu_q = cu_q; job.cu_k = cu_k;
    job.n_seq = n_seq; job.Hq = Hq; job.Hkv = Hkv; job.d = d;
    job.scale = scale;
    job.tokens = tokens; job.heads = heads; job.n_rows = n_rows;
    job.o = o; job.lse = lse;
    for (int32_t s = 0; s < n_seq; ++s) {
        int64_t lk = cu_k[s + 1] - cu_k[s];
        if (lk > job.max_lk)
            job.max_lk = lk;
    }
    pthread_mutex_init(&job.lock, NULL);
    if (n_threads < 1)
        n_threads = 1;
    if (n_threads > 1024)
        n_threads = 1024;
    pthread_t tid[1024];
    int32_t started = 0;
    for (int32_t t = 1; t < n_threads; ++t) {
        if (pthread_create(&tid[started], NULL, row_worker, &job) != 0)
            break;
        ++started;
    }
    row_worker(&job);
    for (int32_t t = 0; t < started; ++t)
        pthread_join(tid[t], NULL);
    pthread_mutex_destroy(&job.lock);
    return job.failed ? -1 : 0;
}

/* Every row: o is [total_q, Hq, d] doubles, lse is [total_q, Hq] doubles. */
int oracle_attention(const uint16_t *q, const uint16_t *k, const uint16_t *v,
                     const int32_t *cu_q, const int32_t *cu_k, int32_t n_seq,
                     int32_t Hq, int32_t Hkv, int32_t d, double scale,
                     double *o, double *lse, int32_t n_threads)
{
    if (n_seq < 0 || Hq <= 0)
        return -1;
    int64_t total_q = cu_q[n_seq];
    int64_t n_rows = total_q * Hq;
    int64_t *tokens = (int64_t *)malloc(sizeof(int64_t) * (size_t)(n_rows > 0 ? n_rows : 1));
    int32_t *heads = (int32_t *)malloc(sizeof(int32_t) * (size_t)(n_rows > 0 ? n_rows : 1));
    if (!tokens || !heads) {
        free(tokens);
        free(heads);
        return -1;
    }
    for (int64_t t = 0; t < total_q; ++t)
        for (int32_t h = 0; h < Hq; ++h) {
            tokens[t * Hq + h] = t;
            heads[t * Hq + h] = h;
        }
    int rc = oracle_attention_rows(q, k, v, cu_q, cu_k, n_seq, Hq, Hkv, d, scale,
                                   tokens, heads, n_rows, o, lse, n_threads);
    free(tokens);
    free(heads);
    return rc;
}
