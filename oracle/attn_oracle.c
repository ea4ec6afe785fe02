/*
 * RefAdapt-DiT CPU oracle: joint attention by its plain definition, in fp64.
 *
 * TEST INFRASTRUCTURE ONLY. This file is compiled into oracle/liboracle.so and
 * is called only by the test suite, by __graft_entry__.smoke() and by the
 * cpu_baseline / reference legs of bench.py. The product library never links
 * it, and it shares no code, header or constant with the CUDA path.
 *
 * What it computes (paper Sec. 3.3, the attention operator
 * Attn(Q,K,V) = Softmax(Q K^T / sqrt(d_h)) V, and Eq. 4, the directional
 * exposure):
 *
 *   for every head h and every query row i:
 *     s_j   = scale * <q_i, k_j>  (+ beta_h when row i is a target row and
 *                                   key j lies in the reference range [r0, r1))
 *     p_j   = exp(s_j - max_l s_l) / sum_l exp(s_l - max_l s_l)
 *     o_i   = sum_j p_j v_j
 *     mass_i = sum_{j in [r0, r1)} p_j          (inner sum of Eq. 4)
 *
 * The outer mean of Eq. 4 over target rows is taken by the Python side.
 * No online softmax, no tiling, no blocking: one row at a time, all keys at
 * once. Rows are split across plain pthreads; each row is computed by exactly
 * one thread in a fixed order, so the result does not depend on the thread
 * count.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>

typedef struct {
    int64_t H, nq, nk, d;
    const double *q, *k, *v;
    double scale;
    const double *bias;          /* [H] or NULL */
    const uint8_t *row_biased;   /* [nq] or NULL: rows that receive the bias */
    int64_t r0, r1;              /* reference key range */
    double *o;                   /* [H][nq][d] */
    double *mass;                /* [H][nq] */
    int64_t first, stride;       /* this worker's share of (h, i) pairs */
    int status;
} oracle_job;

static void *oracle_worker(void *arg)
{
    oracle_job *J = (oracle_job *)arg;
    double *s = (double *)malloc(sizeof(double) * (size_t)(J->nk > 0 ? J->nk : 1));
    if (!s) { J->status = -1; return NULL; }
    const int64_t total = J->H * J->nq;
    for (int64_t w = J->first; w < total; w += J->stride) {
        const int64_t h = w / J->nq;
        const int64_t i = w % J->nq;
        const double *qi = J->q + (h * J->nq + i) * J->d;
        const double *kh = J->k + h * J->nk * J->d;
        const double *vh = J->v + h * J->nk * J->d;
        const int biased = J->bias && J->row_biased && J->row_biased[i];
        /* logits */
        double smax = -INFINITY;
        for (int64_t j = 0; j < J->nk; ++j) {
            double dot = 0.0;
            for (int64_t c = 0; c < J->d; ++c) dot += qi[c] * kh[j * J->d + c];
            double sj = J->scale * dot;
            if (biased && j >= J->r0 && j < J->r1) sj += J->bias[h];
            s[j] = sj;
            if (sj > smax) smax = sj;
        }
        /* normaliser */
        double z = 0.0;
        for (int64_t j = 0; j < J->nk; ++j) { s[j] = exp(s[j] - smax); z += s[j]; }
        /* probabilities, output row (skipped when o is NULL) and reference mass */
        double *oi = J->o ? J->o + (h * J->nq + i) * J->d : NULL;
        if (oi) for (int64_t c = 0; c < J->d; ++c) oi[c] = 0.0;
        double m = 0.0;
        for (int64_t j = 0; j < J->nk; ++j) {
            const double p = s[j] / z;
            if (j >= J->r0 && j < J->r1) m += p;
            if (oi) for (int64_t c = 0; c < J->d; ++c) oi[c] += p * vh[j * J->d + c];
        }
        J->mass[h * J->nq + i] = m;
    }
    free(s);
    J->status = 0;
    return NULL;
}

/*
 * q: [H][nq][d], k, v: [H][nk][d], o: [H][nq][d] (may be NULL: mass only),
 * mass: [H][nq]; all fp64, contiguous. Returns 0 on success, -1 on bad
 * arguments or allocation failure.
 */
int oracle_joint_attn_f64(int64_t H, int64_t nq, int64_t nk, int64_t d,
                          const double *q, const double *k, const double *v,
                          double scale, const double *bias, const uint8_t *row_biased,
                          int64_t r0, int64_t r1, double *o, double *mass, int nthreads)
{
    if (H < 0 || nq < 0 || nk <= 0 || d <= 0 || r0 < 0 || r1 < r0 || r1 > nk) return -1;
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 1024) nthreads = 1024;
    oracle_job *jobs = (oracle_job *)calloc((size_t)nthreads, sizeof(oracle_job));
    pthread_t *tids = (pthread_t *)calloc((size_t)nthreads, sizeof(pthread_t));
    if (!jobs || !tids) { free(jobs); free(tids); return -1; }
    int started = 0, rc = 0;
    for (int t = 0; t < nthreads; ++t) {
        oracle_job J = {H, nq, nk, d, q, k, v, scale, bias, row_biased, r0, r1, o, mass,
                        t, nthreads, 0};
        jobs[t] = J;
    }
    for (int t = 1; t < nthreads; ++t) {
        if (pthread_create(&tids[t], NULL, oracle_worker, &jobs[t]) != 0) { rc = -1; break; }
        ++started;
    }
    if (rc != 0) {
        /* fall back to running the remaining shares on this thread */
        for (int t = started + 1; t < nthreads; ++t) oracle_worker(&jobs[t]);
        rc = 0;
    }
    oracle_worker(&jobs[0]);
    for (int t = 1; t <= started; ++t) pthread_join(tids[t], NULL);
    for (int t = 0; t < nthreads; ++t) if (jobs[t].status != 0) rc = -1;
    free(jobs);
    free(tids);
    return rc == 0 ? 0 : -1;
}
