/*
 * Oracle: causal replay attention by its plain definition, in fp64.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file or the library built from it; only the tests, the smoke
 * check and the benchmark's CPU-baseline leg use it.  It shares no code with
 * the CUDA library.
 *
 * What it computes (Alg. 1, replay loop R <- F(R, o_t); the suffix is
 * re-materialised by prefill on the cropped cache, Sec. 3.2):
 *   the cache of one sequence holds n_keys tokens; the n_q queries are the
 *   LAST n_q positions (bottom-right causal alignment), so query i sits at
 *   absolute position a = n_keys - n_q + i and sees keys j = 0..a.
 *   For q-head h the key/value head is h / (hq / hkv) (consecutive groups).
 *     s_j = scale * sum_c q[c] * K_j[c]
 *     m   = max_j s_j
 *     w_j = exp(s_j - m)
 *     O   = sum_j w_j V_j / sum_j w_j
 * Inputs are bf16 bit patterns, decoded exactly to double; every sum runs in
 * ascending index order in double precision, so one row's result does not
 * depend on which other rows are computed (this is what makes the splice
 * check of Theorem 1 an exact equality).
 *
 * Work is spread over threads by (row, head) item; each item's arithmetic is
 * the same whatever thread runs it.
 */
#include <math.h>
#include <pthread.h>
#include <stdatomic.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <unistd.h>

static double bf16_value(uint16_t bits)
{
    uint32_t u = (uint32_t)bits << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

typedef struct {
    const uint16_t *q, *k, *v;
    int64_t n_q, n_keys;
    int32_t hq, hkv, d;
    double scale;
    const int64_t *rows;
    int64_t n_rows;
    double *out;
    atomic_llong next;
    atomic_int failed;
} job_t;

static int one_item(job_t *jb, int64_t item, double *scores)
{
    const int64_t r = item / jb->hq;
    const int32_t h = (int32_t)(item % jb->hq);
    const int64_t i = jb->rows ? jb->rows[r] : r;
    const int32_t d = jb->d;
    const int32_t group = jb->hq / jb->hkv;
    const int32_t kvh = h / group;
    const int64_t a = jb->n_keys - jb->n_q + i; /* absolute position of query i */
    const uint16_t *qrow = jb->q + (i * jb->hq + h) * (int64_t)d;
    double *o = jb->out + (r * jb->hq + h) * (int64_t)d;

    double m = -INFINITY;
    for (int64_t j = 0; j <= a; ++j) {
        const uint16_t *krow = jb->k + (j * jb->hkv + kvh) * (int64_t)d;
        double s = 0.0;
        for (int32_t c = 0; c < d; ++c)
            s += bf16_value(qrow[c]) * bf16_value(krow[c]);
        s *= jb->scale;
        scores[j] = s;
        if (s > m)
            m = s;
    }
    double den = 0.0;
    for (int32_t c = 0; c < d; ++c)
        o[c] = 0.0;
    for (int64_t j = 0; j <= a; ++j) {
        const double w = exp(scores[j] - m);
        const uint16_t *vrow = jb->v + (j * jb->hkv + kvh) * (int64_t)d;
        den += w;
        for (int32_t c = 0; c < d; ++c)
            o[c] += w * bf16_value(vrow[c]);
    }
    for (int32_t c = 0; c < d; ++c)
        o[c] /= den;
    return 0;
}

static void *worker(void *arg)
{
    job_t *jb = (job_t *)arg;
    double *scores = (double *)malloc(sizeof(double) * (size_t)(jb->n_keys > 0 ? jb->n_keys : 1));
    if (!scores) {
        atomic_store(&jb->failed, 1);
        return NULL;
    }
    const int64_t total = jb->n_rows * jb->hq;
    for (;;) {
        const int64_t item = atomic_fetch_add(&jb->next, 1);
        if (item >= total)
            break;
        one_item(jb, item, scores);
    }
    free(scores);
    return NULL;
}

int oracle_num_cpus(void)
{
    long n = sysconf(_SC_NPROCESSORS_ONLN);
    return n > 0 ? (int)n : 1;
}

/*
 * q   : bf16 bits [n_q][hq][d]
 * k, v: bf16 bits [n_keys][hkv][d]   (the sequence's keys in logical order)
 * rows: query indices to compute (NULL = all n_q, in order)
 * out : fp64 [n_rows][hq][d]
 * Returns 0, or -1 on invalid arguments / allocation failure.
 */
int oracle_causal_attention(const uint16_t *q, int64_t n_q, const uint16_t *k, const uint16_t *v,
                            int64_t n_keys, int32_t hq, int32_t hkv, int32_t d, double scale,
                            const int64_t *rows, int64_t n_rows, double *out, int32_t nthreads)
{
    if (n_q < 0 || n_keys < 0 || n_q > n_keys || hq <= 0 || hkv <= 0 || d <= 0 || hq % hkv != 0)
        return -1;
    if (!rows)
        n_rows = n_q;
    for (int64_t r = 0; rows && r < n_rows; ++r)
        if (rows[r] < 0 || rows[r] >= n_q)
            return -1;
    if (n_rows == 0)
        return 0;

    job_t jb;
    jb.q = q; jb.k = k; jb.v = v;
    jb.n_q = n_q; jb.n_keys = n_keys;
    jb.hq = hq; jb.hkv = hkv; jb.d = d;
    jb.scale = scale;
    jb.rows = rows; jb.n_rows = n_rows;
    jb.out = out;
    atomic_init(&jb.next, 0);
    atomic_init(&jb.failed, 0);

    if (nthreads <= 0)
        nthreads = oracle_num_cpus();
    const int64_t items = n_rows * hq;
    if (nthreads > items)
        nthreads = (int32_t)items;
    if (nthreads <= 1) {
        worker(&jb);
    } else {
        pthread_t *th = (pthread_t *)malloc(sizeof(pthread_t) * (size_t)nthreads);
        if (!th)
            return -1;
        int started = 0;
        for (int t = 0; t < nthreads; ++t) {
            if (pthread_create(&th[t], NULL, worker, &jb) != 0)
                break;
            ++started;
        }
        if (started == 0)
            worker(&jb);
        for (int t = 0; t < started; ++t)
            pthread_join(th[t], NULL);
        free(th);
    }
    return atomic_load(&jb.failed) ? -1 : 0;
}
