/*
 * All-cores variant of litevlm_oracle_score (litevlm_oracle.c), for the
 * benchmark's CPU baseline.
 *
 * TEST INFRASTRUCTURE ONLY, like the rest of this directory: the benchmark's
 * CPU-baseline and reference legs and the tests load it; the CUDA path never
 * does.
 *
 * Same definition and readings as litevlm_oracle_score (Design section, Token
 * Selection Module; the oracle's header lists them): every text query i of
 * head h gives a softmax row P[h][i][:] over the request's visual tokens, and
 * score[j] = (sum_h sum_i P[h][i][j]) / (Hq * T_b). The work is spread over
 * POSIX threads without changing a single rounding:
 *   1. the (h, i) rows are independent: each thread computes whole rows (the
 *      dot products in ascending c, the maximum, the sum of exponentials in
 *      ascending j, then every P[h][i][j]) exactly as the serial loop does,
 *      and stores P;
 *   2. the visual tokens are independent: each thread takes a range of j and
 *      adds P[h][i][j] over the rows in the serial order (h outer, i inner),
 *      starting from 0.0 as the serial accumulator does.
 * So the scores equal the serial oracle's bit for bit (a test checks it).
 * Memory: one request's P, Hq * T_b * N_b doubles, at a time.
 */
#define _POSIX_C_SOURCE 200809L
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>

double litevlm_oracle_decode(int32_t dtype, const void* base, int64_t index);

#define ORT_MAX_THREADS 256

typedef struct {
    /* the request */
    const double* qd;  /* [tb][hq][d] */
    const double* kd;  /* [nb][hkv][d] */
    double* P;         /* [hq * tb][nb] */
    double* acc;       /* [nb] */
    int64_t nb, tb;
    int32_t hq, hkv, d, group;
    double scale;
    /* this worker's share */
    int64_t begin, end;
} ort_job;

static void* ort_rows(void* arg)
{
    const ort_job* J = (const ort_job*)arg;
    for (int64_t row = J->begin; row < J->end; ++row) {
        const int32_t h = (int32_t)(row / J->tb);
        const int64_t i = row - (int64_t)h * J->tb;
        const int32_t g = h / J->group;
        const int64_t qrow = (i * J->hq + h) * J->d;
        double* p = J->P + row * J->nb;
        double m = -INFINITY, l = 0.0;
        for (int64_t j = 0; j < J->nb; ++j) {
            const int64_t krow = (j * J->hkv + g) * J->d;
            double dot = 0.0;
            for (int32_t c = 0; c < J->d; ++c) dot += J->qd[qrow + c] * J->kd[krow + c];
            p[j] = dot * J->scale;  /* the logit, overwritten by P below */
            if (p[j] > m) m = p[j];
        }
        for (int64_t j = 0; j < J->nb; ++j) l += exp(p[j] - m);
        for (int64_t j = 0; j < J->nb; ++j) p[j] = exp(p[j] - m) / l;
    }
    return NULL;
}

static void* ort_cols(void* arg)
{
    const ort_job* J = (const ort_job*)arg;
    const int64_t rows = (int64_t)J->hq * J->tb;
    for (int64_t j = J->begin; j < J->end; ++j) {
        double a = 0.0;
        for (int64_t row = 0; row < rows; ++row) a += J->P[row * J->nb + j];
        J->acc[j] = a;
    }
    return NULL;
}

/* Runs fn over [0, n) split into `threads` contiguous ranges. */
static int ort_parallel(void* (*fn)(void*), ort_job* base, int64_t n, int32_t threads)
{
    pthread_t tid[ORT_MAX_THREADS];
    ort_job jobs[ORT_MAX_THREADS];
    int32_t started = 0, rc = 0;
    if (threads > n) threads = (int32_t)(n > 0 ? n : 1);
    for (int32_t t = 0; t < threads; ++t) {
        jobs[t] = *base;
        jobs[t].begin = n * t / threads;
        jobs[t].end = n * (t + 1) / threads;
    }
    for (int32_t t = 1; t < threads; ++t) {
        if (pthread_create(&tid[t], NULL, fn, &jobs[t]) != 0) {
            rc = -1;
            break;
        }
        ++started;
    }
    fn(&jobs[0]);
    for (int32_t t = 1; t <= started; ++t) pthread_join(tid[t], NULL);
    if (rc != 0)  /* a thread could not be started: do its share here */
        for (int32_t t = started + 1; t < threads; ++t) fn(&jobs[t]);
    return 0;
}

/* Arguments and result as litevlm_oracle_score without the optional outputs. */
int litevlm_oracle_score_threads(int32_t batch, const int32_t* seq_offsets, const int32_t* text_offsets,
                                 int32_t hq, int32_t hkv, int32_t head_dim, int32_t dtype,
                                 const void* q, const void* k, double q_scale, double k_scale,
                                 float* scores, int32_t threads)
{
    if (batch < 0 || hq <= 0 || hkv <= 0 || head_dim <= 0 || hq % hkv != 0) return -1;
    if (dtype < 0 || dtype > 2) return -1;
    if (threads < 1) threads = 1;
    if (threads > ORT_MAX_THREADS) threads = ORT_MAX_THREADS;
    for (int32_t b = 0; b < batch; ++b) {
        if (seq_offsets[b + 1] < seq_offsets[b] || text_offsets[b + 1] < text_offsets[b]) return -1;
        if (seq_offsets[b + 1] > seq_offsets[b] && text_offsets[b + 1] == text_offsets[b]) return -1;
    }
    for (int32_t b = 0; b < batch; ++b) {
        const int64_t n0 = seq_offsets[b], nb = seq_offsets[b + 1] - seq_offsets[b];
        const int64_t t0 = text_offsets[b], tb = text_offsets[b + 1] - text_offsets[b];
        if (nb == 0) continue;
        double* qd = (double*)malloc((size_t)(tb * hq * head_dim) * sizeof(double));
        double* kd = (double*)malloc((size_t)(nb * hkv * head_dim) * sizeof(double));
        double* P = (double*)malloc((size_t)(hq * tb * nb) * sizeof(double));
        double* acc = (double*)malloc((size_t)nb * sizeof(double));
        if (!qd || !kd || !P || !acc) {
            free(qd);
            free(kd);
            free(P);
            free(acc);
            return -2;
        }
        for (int64_t x = 0; x < tb * hq * head_dim; ++x) qd[x] = litevlm_oracle_decode(dtype, q, t0 * hq * head_dim + x);
        for (int64_t x = 0; x < nb * hkv * head_dim; ++x) kd[x] = litevlm_oracle_decode(dtype, k, n0 * hkv * head_dim + x);
        ort_job J;
        J.qd = qd;
        J.kd = kd;
        J.P = P;
        J.acc = acc;
        J.nb = nb;
        J.tb = tb;
        J.hq = hq;
        J.hkv = hkv;
        J.d = head_dim;
        J.group = hq / hkv;
        J.scale = q_scale * k_scale / sqrt((double)head_dim);
        ort_parallel(ort_rows, &J, (int64_t)hq * tb, threads);
        ort_parallel(ort_cols, &J, nb, threads);
        const double denom = (double)hq * (double)tb;
        for (int64_t j = 0; j < nb; ++j) scores[n0 + j] = (float)(acc[j] / denom);
        free(qd);
        free(kd);
        free(P);
        free(acc);
    }
    return 0;
}
