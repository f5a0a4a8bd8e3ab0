/*
 * CPU oracle: decode attention over one sequence's KV rows.
 *
 * TEST INFRASTRUCTURE ONLY.  Only tests/, __graft_entry__.smoke() and
 * bench.py's CPU-baseline / reference legs may load this library.  The CUDA
 * path shares no code, header, table or constant with it.
 *
 * What it computes (Sec. 1 and Sec. 3.4: decoding one token attends over the
 * whole KV cache; Sec. 2.1: grouped-query attention shares one K/V head among
 * a group of query heads).  The paper prints no formula; this is the textbook
 * scaled-dot-product decode for one query token:
 *
 *   for query head h, KV head g = floor(h / G), G = Hq / Hkv:
 *     s_t  = scale * sum_e q[h][e] * K[t][g][e]        t = 0 .. n-1
 *     m    = max_t s_t
 *     p_t  = exp(s_t - m)
 *     l    = sum_t p_t
 *     o[h] = (sum_t p_t * V[t][g][:]) / l
 *
 * Inputs are bf16 bit patterns, widened exactly to double; all arithmetic is
 * double, summed sequentially over t in logical order (two passes).
 * An optional mask (mask[t] != 0) removes token t from the softmax: its
 * weight is exactly zero (Sec. 3.3 / Algorithm 2, BuildMask: masking a closed
 * cursor's tokens stands for having evicted them).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

static double widen_bf16(uint16_t bits) {
    uint32_t u = ((uint32_t)bits) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* One query head.  k, v: [n][Hkv][d] bf16 bits.  Returns 0, or -1 when every
 * token is masked or n == 0. */
static int one_head(int n, int Hkv, int d, int g, const uint16_t *qh,
                    const uint16_t *k, const uint16_t *v, double scale,
                    const uint8_t *mask, double *out, double *weights,
                    double *lse) {
    double *s = (double *)malloc(sizeof(double) * (size_t)(n > 0 ? n : 1));
    double *qd = (double *)malloc(sizeof(double) * (size_t)d);
    if (!s || !qd) { free(s); free(qd); return -2; }
    for (int e = 0; e < d; ++e) qd[e] = widen_bf16(qh[e]);

    /* pass 1: logits and their maximum */
    double m = -INFINITY;
    int any = 0;
    for (int t = 0; t < n; ++t) {
        if (mask && mask[t]) { s[t] = -INFINITY; continue; }
        const uint16_t *kt = k + ((size_t)t * Hkv + g) * d;
        double acc = 0.0;
        for (int e = 0; e < d; ++e) acc += qd[e] * widen_bf16(kt[e]);
        s[t] = scale * acc;
        if (s[t] > m) m = s[t];
        any = 1;
    }
    if (!any) { free(s); free(qd); return -1; }

    /* pass 2: exponentials, their sum and the weighted sum of V */
    for (int e = 0; e < d; ++e) out[e] = 0.0;
    double l = 0.0;
    for (int t = 0; t < n; ++t) {
        if (mask && mask[t]) { s[t] = 0.0; continue; }
        double p = exp(s[t] - m);
        s[t] = p;
        l += p;
        const uint16_t *vt = v + ((size_t)t * Hkv + g) * d;
        for (int e = 0; e < d; ++e) out[e] += p * widen_bf16(vt[e]);
    }
    for (int e = 0; e < d; ++e) out[e] /= l;
    if (weights)
        for (int t = 0; t < n; ++t) weights[t] = s[t] / l;
    if (lse) *lse = m + log(l);
    free(s);
    free(qd);
    return 0;
}

/*
 * Decode attention of one sequence for all query heads.
 *   q:   [Hq][d]        bf16 bits
 *   k,v: [n][Hkv][d]    bf16 bits (logical token order)
 *   mask: [n] or NULL
 *   out: [Hq][d]        double
 *   weights: [Hq][n] or NULL (normalised softmax weights)
 *   lse: [Hq] or NULL   (m + log l)
 * Returns 0 on success, -1 on an invalid shape or an all-masked row.
 */
int oracle_decode_f64(int n, int Hq, int Hkv, int d, const uint16_t *q,
                      const uint16_t *k, const uint16_t *v, double scale,
                      const uint8_t *mask, double *out, double *weights,
                      double *lse) {
    if (n <= 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || Hq % Hkv != 0) return -1;
    int G = Hq / Hkv;
    int status = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(min : status)
    for (int h = 0; h < Hq; ++h) {
        int rc = one_head(n, Hkv, d, h / G, q + (size_t)h * d, k, v, scale,
                          mask, out + (size_t)h * d,
                          weights ? weights + (size_t)h * n : NULL,
                          lse ? lse + h : NULL);
        if (rc < status) status = rc;
    }
    return status;
}

/*
 * The same for a batch of independent sequences (one decode step of a
 * batch): OpenMP over (sequence, query head) pairs.
 *   ns[i]            token count of sequence i
 *   q  + i*Hq*d      its query
 *   ks[i], vs[i]     its [ns[i]][Hkv][d] rows
 *   out + i*Hq*d     its output
 */
int oracle_decode_batch_f64(int n_seqs, const int *ns, int Hq, int Hkv, int d,
                            const uint16_t *q, const uint16_t *const *ks,
                            const uint16_t *const *vs, double scale,
                            double *out) {
    if (n_seqs < 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || Hq % Hkv != 0) return -1;
    int G = Hq / Hkv;
    int status = 0;
    long total = (long)n_seqs * Hq;
#pragma omp parallel for schedule(dynamic, 1) reduction(min : status)
    for (long w = 0; w < total; ++w) {
        int i = (int)(w / Hq), h = (int)(w % Hq);
        int rc = ns[i] > 0
                     ? one_head(ns[i], Hkv, d, h / G,
                                q + ((size_t)i * Hq + h) * d, ks[i], vs[i],
                                scale, NULL, out + ((size_t)i * Hq + h) * d,
                                NULL, NULL)
                     : -1;
        if (rc < status) status = rc;
    }
    return status;
}

/*
 * Quantities for the error analysis of a decode whose softmax weights each
 * carry a small relative perturbation (for instance weights rounded to a
 * narrower type before the PV product).  Not part of the method: the tests
 * build their error budgets from them.  For query head h, KV head
 * g = floor(h / G) and every dimension e, with w_t the exact softmax weights
 * and o[h] the exact output (both exactly as oracle_decode_f64 computes them):
 *   dev[h][e]  = sum_t w_t * |V[t][g][e] - o[h][e]|
 *   absv[h][e] = sum_t w_t * |V[t][g][e]|
 * out receives o.  Same shapes and return codes as oracle_decode_f64.
 */
int oracle_decode_dev_f64(int n, int Hq, int Hkv, int d, const uint16_t *q,
                          const uint16_t *k, const uint16_t *v, double scale,
                          const uint8_t *mask, double *out, double *dev,
                          double *absv) {
    if (n <= 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || Hq % Hkv != 0) return -1;
    int G = Hq / Hkv;
    int status = 0;
#pragma omp parallel for schedule(dynamic, 1) reduction(min : status)
    for (int h = 0; h < Hq; ++h) {
        double *w = (double *)malloc(sizeof(double) * (size_t)n);
        if (!w) { status = -2; continue; }
        const int g = h / G;
        double *o = out + (size_t)h * d;
        int rc = one_head(n, Hkv, d, g, q + (size_t)h * d, k, v, scale, mask, o, w,
                          NULL);
        if (rc == 0) {
            double *dv = dev + (size_t)h * d, *av = absv + (size_t)h * d;
            for (int e = 0; e < d; ++e) { dv[e] = 0.0; av[e] = 0.0; }
            for (int t = 0; t < n; ++t) {
                if (w[t] == 0.0) continue;
                const uint16_t *vt = v + ((size_t)t * Hkv + g) * d;
                for (int e = 0; e < d; ++e) {
                    const double x = widen_bf16(vt[e]);
                    dv[e] += w[t] * fabs(x - o[e]);
                    av[e] += w[t] * fabs(x);
                }
            }
        }
        free(w);
        if (rc < status) status = rc;
    }
    return status;
}

/*
 * Masked prefill attention (Algorithm 2, BuildMask; Sec. 3.3: the auxiliary
 * training traces see the context with the closed cursors' tokens masked
 * out).  The last n_q tokens of a sequence of n tokens are the queries; query
 * i sits at logical position p = n - n_q + i and attends to the tokens
 * t = 0 .. p (causal) that are not removed (removed[t] != 0).  Per query and
 * head this is exactly the decode above over the rows 0 .. p with the
 * removal mask.  A query that sees no token gets a zero output and a log-sum-
 * exp of -infinity (a reading: the paper never masks a whole prefix).
 *   q:   [n_q][Hq][d] bf16 bits       k, v: [n][Hkv][d] bf16 bits
 *   removed: [n] or NULL              out: [n_q][Hq][d] double
 *   lse: [n_q][Hq] or NULL (natural log of sum_t exp(s_t))
 * Returns 0, or -1 on an invalid shape.
 */
int oracle_prefill_f64(int n, int n_q, int Hq, int Hkv, int d, const uint16_t *q,
                       const uint16_t *k, const uint16_t *v, double scale,
                       const uint8_t *removed, double *out, double *lse) {
    if (n <= 0 || n_q <= 0 || n_q > n || Hq <= 0 || Hkv <= 0 || d <= 0 ||
        Hq % Hkv != 0)
        return -1;
    int G = Hq / Hkv;
    int status = 0;
    long total = (long)n_q * Hq;
#pragma omp parallel for schedule(dynamic, 4) reduction(min : status)
    for (long w = 0; w < total; ++w) {
        int i = (int)(w / Hq), h = (int)(w % Hq);
        int p = n - n_q + i;
        double *o = out + ((size_t)i * Hq + h) * d;
        double l_se = 0.0;
        int rc = one_head(p + 1, Hkv, d, h / G, q + ((size_t)i * Hq + h) * d, k, v,
                          scale, removed, o, NULL, &l_se);
        if (rc == -1) {  /* every visible token removed */
            for (int e = 0; e < d; ++e) o[e] = 0.0;
            l_se = -INFINITY;
            rc = 0;
        }
        if (lse) lse[(size_t)i * Hq + h] = l_se;
        if (rc < status) status = rc;
    }
    return status;
}

/* Sets the number of OpenMP threads (timing runs only; no effect on results). */
void oracle_set_threads(int n) {
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* Number of OpenMP threads the two entry points above run with. */
int oracle_num_threads(void) {
    int n = 1;
#ifdef _OPENMP
#pragma omp parallel
    {
#pragma omp single
        n = omp_get_num_threads();
    }
#endif
    return n;
}
