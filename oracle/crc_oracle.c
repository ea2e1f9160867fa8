/*
 * Plain CPU oracle for cache-aware MoE routing and expert residency.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may link, load or
 * call this file; only the tests, the smoke check and the benchmark's timed
 * CPU baseline do.  It shares no code with the CUDA library.
 *
 * What it computes, step by step, in the paper's order and notation
 * ("Cache-Aware Joint Router Adaptation for Memory-Efficient MoE Inference"):
 *
 *   router heads   p^X_{t,l} = softmax(W^X_l h_{t,l}),  X in {R, T, S}
 *                  (Sec. 2 problem statement; Sec. 3.2 Temporal head;
 *                  Sec. 3.3 Spatio head).  Dot products and softmax in fp64
 *                  from the bf16 inputs; softmax as exp(z - max z) / sum.
 *   native Top-K   S_{t,l} = TopK(p^R_{t,l})                       (Sec. 2)
 *   retention      s^T_{t,l} = p^R_{t,l} + p^T_{t,l}               (Sec. 3.2)
 *                  C_{t+1,l} = UpdateCache(C~, S, s^T, C)          (Algorithm 1)
 *   refinement     a^T_{t,l} = p^R_{t-1,l} + p^T_{t-1,l}
 *                  s^ST_{t,l} = a^T_{t,l} + p^S_{rho(t,l)}         (Sec. 3.3)
 *                  rho(t,1) = (t-1, L), rho(t,l) = (t, l-1)
 *                  top-R candidates, insert / replace-lowest        (Algorithm 2)
 *   accounting     accesses, demand misses D, proactive loads P   (Sec. 4.1)
 *
 * Readings where the paper is silent (each one is listed in the design notes):
 *   - one total order everywhere: score descending, expert index ascending.
 *     TopK / Top_R take its first elements; every argmin takes its LAST
 *     element, i.e. the smallest score and, among equal scores, the highest
 *     expert index;
 *   - the refinement test is strict (a candidate must be strictly higher);
 *   - Top_R ranges over all N experts, residents included (residents are
 *     skipped), so P <= R per access;
 *   - no refinement at the first token (t = 0) of any layer: there is no
 *     previous-token state a^T yet;
 *   - caches start empty (cold start) and every token is counted;
 *   - the demand set D of Algorithm 1 is walked in ascending expert index.
 *
 * Two precisions of the cache scan are built from one body: fp64 (the
 * end-to-end oracle, fed by fp64 router probabilities) and fp32 (the scan fed
 * with fp32 probabilities, taking every sum and comparison in fp32 as the
 * kernel does: s^T = fp32(p^R + p^T), s^ST = fp32(fp32(a^T) + p^S)).
 *
 * Layouts (row-major): hidden bf16 bits [B][T][L][d]; weights bf16 bits
 * [L][3N][d] with heads ordered R, T, S; probabilities [B][T][L][3][N].
 * Layers and tokens are 0-indexed here, so rho(t,0) = (t-1, L-1).
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_MAX_N 256

/* ------------------------------------------------------------------------ */
/* router probabilities                                                      */
/* ------------------------------------------------------------------------ */
static double bf16_to_double(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* One unit: H heads of N probabilities each, from one hidden row and the
 * weight block of its layer ([3N][d], only the first H*N rows are read). */
void oracle_unit_probs(int N, int d, int H, const uint16_t *h_row,
                       const uint16_t *w_layer, double *out /* [H][N] */)
{
    double hv[8192];
    double *hbuf = hv;
    if (d > 8192) hbuf = (double *)malloc(sizeof(double) * (size_t)d);
    for (int i = 0; i < d; i++) hbuf[i] = bf16_to_double(h_row[i]);
    double z[ORACLE_MAX_N];
    for (int head = 0; head < H; head++) {
        for (int e = 0; e < N; e++) {
            const uint16_t *w = w_layer + ((size_t)head * N + e) * d;
            double acc = 0.0;
            for (int i = 0; i < d; i++) acc += bf16_to_double(w[i]) * hbuf[i];
            z[e] = acc;
        }
        double zmax = z[0];
        for (int e = 1; e < N; e++)
            if (z[e] > zmax) zmax = z[e];
        double sum = 0.0;
        for (int e = 0; e < N; e++) {
            z[e] = exp(z[e] - zmax);
            sum += z[e];
        }
        for (int e = 0; e < N; e++) out[head * N + e] = z[e] / sum;
    }
    if (hbuf != hv) free(hbuf);
}

typedef struct {
    int B, T, L, N, d, H;
    const uint16_t *hidden, *w;
    double *probs;
    int64_t begin, end;
} probs_job;

static void *probs_worker(void *arg)
{
    probs_job *j = (probs_job *)arg;
    for (int64_t u = j->begin; u < j->end; u++) {
        int l = (int)(u % j->L);
        oracle_unit_probs(j->N, j->d, j->H, j->hidden + (size_t)u * j->d,
                          j->w + (size_t)l * 3 * j->N * j->d,
                          j->probs + (size_t)u * 3 * j->N);
    }
    return NULL;
}

/* probs [B][T][L][3][N]; heads >= H are left untouched. */
void oracle_router_probs(int B, int T, int L, int N, int d, int H,
                         const uint16_t *hidden, const uint16_t *w_cat,
                         double *probs, int nthreads)
{
    int64_t U = (int64_t)B * T * L;
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    pthread_t th[256];
    probs_job jobs[256];
    int64_t per = (U + nthreads - 1) / nthreads;
    int started = 0;
    for (int k = 0; k < nthreads; k++) {
        probs_job j = {B, T, L, N, d, H, hidden, w_cat, probs,
                       k * per, (k + 1) * per < U ? (k + 1) * per : U};
        jobs[k] = j;
        if (j.begin >= j.end) continue;
        if (nthreads == 1) {
            probs_worker(&jobs[k]);
        } else {
            pthread_create(&th[k], NULL, probs_worker, &jobs[k]);
            started = k + 1;
        }
    }
    for (int k = 0; k < started; k++)
        if (jobs[k].begin < jobs[k].end) pthread_join(th[k], NULL);
}

/* ------------------------------------------------------------------------ */
/* cache scan, one body for two precisions                                   */
/* ------------------------------------------------------------------------ */
static double rel_gap(double a, double b)
{
    double m = fabs(a) > fabs(b) ? fabs(a) : fabs(b);
    if (m == 0.0) return 0.0;
    return fabs(a - b) / m;
}

#define REAL double
#define SFX f64
#include "scan_body.h"
#undef REAL
#undef SFX

#define REAL float
#define SFX f32
#include "scan_body.h"
#undef REAL
#undef SFX

/* ------------------------------------------------------------------------ */
/* reporting (Sec. 4.1 Metrics)                                              */
/* ------------------------------------------------------------------------ */
/* Exposed expert-loading cost per decode token under the overlap model of the
 * appendix on asynchronous transfer overlap: demand transfers fully exposed, a
 * fraction eta of proactive transfer time hidden, c_exp seconds per expert:
 * t_load(eta) = c_exp / T * (D + (1 - eta) * P). */
double oracle_load_time(double D, double P, double T, double c_exp, double eta)
{
    return c_exp / T * (D + (1.0 - eta) * P);
}

/* Hit = 1 - D/A, AdjHit = (A - D)/(A + P), Load/token = (D + P) * S_exp / T. */
void oracle_metrics(double A, double D, double P, double T, double s_exp,
                    double *hit, double *adj_hit, double *load_per_token)
{
    *hit = 1.0 - D / A;
    *adj_hit = (A - D) / (A + P);
    *load_per_token = (D + P) * s_exp / T;
}
