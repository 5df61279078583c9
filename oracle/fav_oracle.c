/*
 * fav_oracle.c -- the fp64 CPU oracle for exact attention.  TEST INFRASTRUCTURE ONLY.
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline / reference leg may
 * load this code.  It shares nothing with the CUDA path (no header, helper or table).
 *
 * What it computes is the plain definition of scaled dot-product attention
 * (FlashAttention-V paper, Background section: Attention(Q,K,V) = softmax(Q K^T / sqrt(D)) V,
 * with the per-head N x D shapes of the Method section, "FlashAttention-V Optimizations"),
 * written out per query row in fp64:
 *
 *   s_j  = scale * sum_d Q[b,h,i,d] * K[b,g,j,d]        for every visible key j
 *   m    = max_j s_j
 *   l    = sum_j exp(s_j - m)
 *   O    = sum_j exp(s_j - m) * V[b,g,j,:] / l
 *   LSE  = m + ln l
 *
 * Readings of points the paper leaves open:
 *  - g = h / (Hq / Hkv): consecutive query heads share one K/V head (Method section on GQA,
 *    where one loaded K row is replicated over the adjacent head slots of a register).
 *  - causal masking (Algorithm "ggml-vec FlashAttention" and Algorithm "FlashAttention-V for
 *    VL > D" both only say "check for causal masking") is bottom-right aligned: query i sits at
 *    position Nkv - Nq + i and sees keys j <= Nkv - Nq + i.  causal with Nq > Nkv is rejected,
 *    so no row is ever empty.
 *  - scale is an explicit argument (the algorithms use an opaque "scale"); callers pass 1/sqrt(D).
 *  - LSE is the natural-log log-sum-exp of the scaled scores (not in the paper).
 *
 * The two passes (max first, then exponentials) are the standard exact evaluation of the
 * softmax; they change no value of the definition, only keep exp() finite.
 * Rows are distributed over POSIX threads; every row is computed by the same scalar loops.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <pthread.h>
#include <stdatomic.h>

typedef struct {
    const double *q, *k, *v;
    double *o, *lse;
    int64_t B, Hq, Hkv, Nq, Nkv, D;
    double scale;
    int causal;
    const int64_t *rows;   /* NULL: every row; else flat indices into [B, Hq, Nq] */
    int64_t nrows;
    double *probs;         /* optional [B, Hq, Nq, Nkv] softmax weights (tiny cases) */
    atomic_llong next;
} job_t;

/* Number of keys row i may see (definition above). */
static int64_t visible_keys(const job_t *J, int64_t i) {
    if (!J->causal) return J->Nkv;
    return J->Nkv - J->Nq + i + 1;
}

/* One query row: two passes over the visible keys, all in fp64. */
static void one_row(const job_t *J, int64_t flat, double *o_out, double *lse_out, double *s) {
    const int64_t D = J->D, Nq = J->Nq, Nkv = J->Nkv;
    const int64_t i = flat % Nq;
    const int64_t h = (flat / Nq) % J->Hq;
    const int64_t b = flat / (Nq * J->Hq);
    const int64_t G = J->Hq / J->Hkv;
    const int64_t g = h / G;
    const double *qr = J->q + flat * D;
    const double *Kh = J->k + (b * J->Hkv + g) * Nkv * D;
    const double *Vh = J->v + (b * J->Hkv + g) * Nkv * D;
    const int64_t n = visible_keys(J, i);

    /* pass 1: scaled scores and their maximum */
    double m = -INFINITY;
    for (int64_t j = 0; j < n; ++j) {
        double dot = 0.0;
        for (int64_t d = 0; d < D; ++d) dot += qr[d] * Kh[j * D + d];
        s[j] = J->scale * dot;
        if (s[j] > m) m = s[j];
    }
    /* pass 2: weights, their sum, and the weighted sum of value rows */
    double l = 0.0;
    for (int64_t d = 0; d < D; ++d) o_out[d] = 0.0;
    for (int64_t j = 0; j < n; ++j) {
        const double w = exp(s[j] - m);
        s[j] = w;
        l += w;
        for (int64_t d = 0; d < D; ++d) o_out[d] += w * Vh[j * D + d];
    }
    for (int64_t d = 0; d < D; ++d) o_out[d] /= l;
    if (lse_out) *lse_out = m + log(l);
    if (J->probs) {
        double *p = J->probs + flat * Nkv;
        for (int64_t j = 0; j < Nkv; ++j) p[j] = (j < n) ? s[j] / l : 0.0;
    }
}

static void *worker(void *arg) {
    job_t *J = (job_t *)arg;
    double *s = (double *)malloc((size_t)(J->Nkv > 0 ? J->Nkv : 1) * sizeof(double));
    if (!s) return (void *)1;
    const int64_t total = J->rows ? J->nrows : J->B * J->Hq * J->Nq;
    for (;;) {
        const int64_t r = (int64_t)atomic_fetch_add(&J->next, 1);
        if (r >= total) break;
        const int64_t flat = J->rows ? J->rows[r] : r;
        double *o_out = J->o + r * J->D;
        double *l_out = J->lse ? J->lse + r : NULL;
        one_row(J, flat, o_out, l_out, s);
    }
    free(s);
    return NULL;
}

static int run(job_t *J, int nthreads) {
    if (!J->q || !J->k || !J->v || !J->o) return 1;
    if (J->B <= 0 || J->Hq <= 0 || J->Hkv <= 0 || J->Nq <= 0 || J->Nkv <= 0 || J->D <= 0) return 1;
    if (J->Hq % J->Hkv != 0) return 1;
    if (J->causal && J->Nq > J->Nkv) return 1;
    if (J->rows) {
        for (int64_t r = 0; r < J->nrows; ++r)
            if (J->rows[r] < 0 || J->rows[r] >= J->B * J->Hq * J->Nq) return 1;
    }
    atomic_init(&J->next, 0);
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 512) nthreads = 512;
    pthread_t th[512];
    int started = 0, err = 0;
    for (int t = 1; t < nthreads; ++t) {
        if (pthread_create(&th[started], NULL, worker, J) != 0) break;
        ++started;
    }
    if (worker(J) != NULL) err = 1;
    for (int t = 0; t < started; ++t) {
        void *ret = NULL;
        pthread_join(th[t], &ret);
        if (ret != NULL) err = 1;
    }
    return err;
}

/* Full forward: o [B,Hq,Nq,D], lse [B,Hq,Nq] (lse may be NULL). Returns 0 on success. */
int fav_oracle_forward(const double *q, const double *k, const double *v, double *o, double *lse,
                       int64_t B, int64_t Hq, int64_t Hkv, int64_t Nq, int64_t Nkv, int64_t D,
                       double scale, int causal, int nthreads) {
    job_t J;
    memset(&J, 0, sizeof(J));
    J.q = q; J.k = k; J.v = v; J.o = o; J.lse = lse;
    J.B = B; J.Hq = Hq; J.Hkv = Hkv; J.Nq = Nq; J.Nkv = Nkv; J.D = D;
    J.scale = scale; J.causal = causal;
    return run(&J, nthreads);
}

/* Selected rows only: rows[r] is a flat index into [B,Hq,Nq]; o [nrows,D], lse [nrows]. */
int fav_oracle_rows(const double *q, const double *k, const double *v,
                    const int64_t *rows, int64_t nrows, double *o, double *lse,
                    int64_t B, int64_t Hq, int64_t Hkv, int64_t Nq, int64_t Nkv, int64_t D,
                    double scale, int causal, int nthreads) {
    if (!rows || nrows < 0) return 1;
    if (nrows == 0) return 0;
    job_t J;
    memset(&J, 0, sizeof(J));
    J.q = q; J.k = k; J.v = v; J.o = o; J.lse = lse;
    J.B = B; J.Hq = Hq; J.Hkv = Hkv; J.Nq = Nq; J.Nkv = Nkv; J.D = D;
    J.scale = scale; J.causal = causal; J.rows = rows; J.nrows = nrows;
    return run(&J, nthreads);
}

/* Full forward that also returns the softmax weights P [B,Hq,Nq,Nkv] (masked keys get 0). */
int fav_oracle_probs(const double *q, const double *k, const double *v, double *o, double *lse,
                     double *probs,
                     int64_t B, int64_t Hq, int64_t Hkv, int64_t Nq, int64_t Nkv, int64_t D,
                     double scale, int causal) {
    if (!probs) return 1;
    job_t J;
    memset(&J, 0, sizeof(J));
    J.q = q; J.k = k; J.v = v; J.o = o; J.lse = lse; J.probs = probs;
    J.B = B; J.Hq = Hq; J.Hkv = Hkv; J.Nq = Nq; J.Nkv = Nkv; J.D = D;
    J.scale = scale; J.causal = causal;
    return run(&J, 1);
}
