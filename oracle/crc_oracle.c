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
 *   coverage loss  m_e = sigmoid((s_e - theta_B(s)) / tau),
 *                  l(s, q) = sum_e q_e (1 - m_e), l^T and l^ST, their means
 *                  and the gradient into the three heads' logits
 *                                                            (Sec. 3.1-3.4)
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
/* Decision margins: the relative gap |a - b| / max(|a|, |b|) between the two
 * scores a decision compares.  A test that builds exact ties on purpose (two
 * experts with identical weight rows have identical scores on every side,
 * and every side breaks such a tie by the same index rule) may exempt gaps of
 * exactly zero; the setting is per thread, made by the scan for its workers. */
static _Thread_local int exact_ties_exempt;

static double rel_gap(double a, double b)
{
    double m = fabs(a) > fabs(b) ? fabs(a) : fabs(b);
    if (a == b && exact_ties_exempt) return INFINITY;
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

/* ------------------------------------------------------------------------ */
/* comparison policies (Sec. 4 baselines "for cache update"; Sec. 4.3 and   */
/* the appendix on ablations for Spatio-only)                               */
/* ------------------------------------------------------------------------ */
/*
 * Readings (the paper names the classical policies and their references and
 * gives LRFU's lambda = 0.5, nothing more):
 *   - the classical policies (LRU, LFU, LRFU) only update the cache: no
 *     pre-access refinement, no proactive load; each access demand-loads
 *     S \ C in ascending expert index and, with the cache full, evicts the
 *     member of V = C \ S with the lowest priority (ties: the highest index),
 *     as Algorithm 1 does with s^T;
 *   - LRU priority: the token index of the expert's last use;
 *   - LFU priority: the number of accesses that selected the expert since it
 *     entered the cache (1 on insertion);
 *   - LRFU priority at token t: CRF * F(t - t_last), CRF updated at each use
 *     to 1 + F(t - t_last) * CRF (1 on insertion), F(x) = 2^(-lambda x) with
 *     lambda a multiple of 1/2, evaluated in fp32 as 2^(-q) (exact), times
 *     fp32(2^(-1/2)) when lambda x is odd in halves, and 0 once q >= 126;
 *   - Spatio-only: Algorithm 2's refinement with s^S = p^R_{t-1} + p^S_rho in
 *     place of s^ST; an expert it loads counts as used at t; the demand loads
 *     evict by LRU.
 */
enum { ORACLE_POLICY_LRU = 1, ORACLE_POLICY_LFU = 2, ORACLE_POLICY_LRFU = 3,
       ORACLE_POLICY_SPATIO_LRU = 4 };

static float lrfu_decay(int lambda2, long dt)        /* F(dt), lambda = lambda2 / 2 */
{
    const long halves = (long)lambda2 * dt;
    const long q = halves / 2;
    if (q >= 126) return 0.0f;
    float f = ldexpf(1.0f, (int)-q);
    if (halves % 2) f = f * 0.70710678118654752f;    /* fp32(2^(-1/2)) */
    return f;
}

/* the member with the smallest integer priority, ties to the highest index */
static int argmin_last_u32(const uint32_t *key, const uint8_t *member, int N)
{
    int v = -1;
    for (int e = 0; e < N; e++)
        if (member[e] && (v < 0 || key[e] <= key[v])) v = e;
    return v;
}

/* One access of one chain under a comparison policy; fp32 throughout. */
int oracle_policy_step(int N, int K, int C, int R, int policy, int lambda2, int t,
                       const float *pR, const float *pS_pred, uint8_t *in_cache, int *count,
                       uint32_t *aux, float *val, int *topk_out, int *misses_out,
                       int *proactive_out)
{
    if (N < 1 || N > ORACLE_MAX_N || K < 1 || K > N || C < K || C > N || R < 0 ||
        policy < ORACLE_POLICY_LRU || policy > ORACLE_POLICY_SPATIO_LRU || lambda2 < 0)
        return -1;
    int proactive = 0;
    /* Spatio-only: pre-access refinement on s^S = p^R_{t-1} + p^S_rho */
    if (policy == ORACLE_POLICY_SPATIO_LRU && R > 0 && t >= 1) {
        float sS[ORACLE_MAX_N];
        uint8_t before[ORACLE_MAX_N];
        for (int e = 0; e < N; e++) {
            sS[e] = val[e] + pS_pred[e];
            before[e] = in_cache[e];
        }
        proactive = oracle_refine_f32(N, C, R, sS, in_cache, count, NULL);
        for (int e = 0; e < N; e++)
            if (in_cache[e] && !before[e]) aux[e] = (uint32_t)t;
    }
    /* native Top-K on p^R */
    int ord[ORACLE_MAX_N];
    order_desc_f32(pR, N, ord);
    uint8_t inS[ORACLE_MAX_N], hit[ORACLE_MAX_N], inV[ORACLE_MAX_N];
    memset(inS, 0, (size_t)N);
    for (int k = 0; k < K; k++) {
        topk_out[k] = ord[k];
        inS[ord[k]] = 1;
    }
    for (int e = 0; e < N; e++) hit[e] = (uint8_t)(inS[e] && in_cache[e]);
    /* the eviction priorities of this access (fixed while it inserts) */
    uint32_t pri_u[ORACLE_MAX_N];
    float pri_f[ORACLE_MAX_N];
    for (int e = 0; e < N; e++) {
        pri_u[e] = aux[e];
        pri_f[e] = policy == ORACLE_POLICY_LRFU ? val[e] * lrfu_decay(lambda2, (long)t - (long)aux[e])
                                                : 0.0f;
    }
    /* demand loads, ascending index; a full cache evicts argmin over C \ S */
    int misses = 0;
    for (int e = 0; e < N; e++) {
        if (!inS[e] || in_cache[e]) continue;
        misses++;
        if (*count < C) {
            in_cache[e] = 1;
            (*count)++;
            continue;
        }
        for (int u = 0; u < N; u++) inV[u] = (uint8_t)(in_cache[u] && !inS[u]);
        int v = policy == ORACLE_POLICY_LRFU ? argmin_last_f32(pri_f, inV, N, NULL)
                                             : argmin_last_u32(pri_u, inV, N);
        in_cache[v] = 0;
        in_cache[e] = 1;
    }
    /* the selected experts' priorities after the access */
    for (int e = 0; e < N; e++) {
        if (!inS[e]) continue;
        if (policy == ORACLE_POLICY_LFU) {
            aux[e] = hit[e] ? aux[e] + 1u : 1u;
        } else if (policy == ORACLE_POLICY_LRFU) {
            val[e] = hit[e] ? 1.0f + lrfu_decay(lambda2, (long)t - (long)aux[e]) * val[e] : 1.0f;
            aux[e] = (uint32_t)t;
        } else {
            aux[e] = (uint32_t)t;
        }
    }
    if (policy == ORACLE_POLICY_SPATIO_LRU)
        for (int e = 0; e < N; e++) val[e] = pR[e];          /* p^R_{t-1} for the next access */
    *misses_out = misses;
    *proactive_out = proactive;
    return 0;
}

/*
 * Whole scan under a comparison policy: B streams, T tokens, L layers, cold
 * start, fp32 probabilities [B][T][L][3][N] (p^S read by Spatio-only only).
 * Outputs as oracle_scan (any trace pointer may be NULL), plus the per-expert
 * policy state of the last token: aux_out [B][L][N] (LRU and Spatio-only:
 * token of last use; LFU: count; LRFU: token of last use) and val_out
 * [B][L][N] (LRFU: CRF; Spatio-only: p^R of the last token; else 0).
 */
int oracle_policy_scan(int B, int T, int L, int N, int K, int C, int R, int policy,
                       int lambda2, const float *probs, uint8_t *topk, uint8_t *misses,
                       uint8_t *proactive, uint32_t *cache_bits, uint32_t *aux_out,
                       float *val_out, uint64_t *counters)
{
    if (B < 0 || T < 0 || L < 1 || N < 1 || N > ORACLE_MAX_N || K < 1 || K > N || C < K ||
        C > N || R < 0)
        return -1;
    const size_t row = (size_t)3 * N;
    uint8_t *in_cache = (uint8_t *)calloc((size_t)L * N, 1);
    int *count = (int *)calloc((size_t)L, sizeof(int));
    uint32_t *aux = (uint32_t *)calloc((size_t)L * N, sizeof(uint32_t));
    float *val = (float *)calloc((size_t)L * N, sizeof(float));
    int tk[ORACLE_MAX_N], rc = 0;
    for (int b = 0; b < B && rc == 0; b++) {
        memset(in_cache, 0, (size_t)L * N);
        memset(count, 0, sizeof(int) * (size_t)L);
        memset(aux, 0, sizeof(uint32_t) * (size_t)L * N);
        memset(val, 0, sizeof(float) * (size_t)L * N);
        uint64_t *ctr = counters + (size_t)b * L * 3;
        memset(ctr, 0, sizeof(uint64_t) * (size_t)L * 3);
        for (int t = 0; t < T && rc == 0; t++) {
            for (int l = 0; l < L; l++) {
                const size_t unit = ((size_t)b * T + t) * L + l;
                const float *pR = probs + unit * row;
                const float *pS = NULL;                     /* p^S_{rho(t,l)} */
                if (l > 0)
                    pS = probs + (unit - 1) * row + 2 * N;
                else if (t > 0)
                    pS = probs + (((size_t)b * T + (t - 1)) * L + (L - 1)) * row + 2 * N;
                int mi, pr;
                if (oracle_policy_step(N, K, C, R, policy, lambda2, t, pR, pS,
                                       in_cache + (size_t)l * N, &count[l], aux + (size_t)l * N,
                                       val + (size_t)l * N, tk, &mi, &pr) != 0) {
                    rc = -1;
                    break;
                }
                ctr[l * 3 + 0] += (uint64_t)(K - mi);
                ctr[l * 3 + 1] += (uint64_t)mi;
                ctr[l * 3 + 2] += (uint64_t)pr;
                if (topk)
                    for (int k = 0; k < K; k++) topk[unit * K + k] = (uint8_t)tk[k];
                if (misses) misses[unit] = (uint8_t)mi;
                if (proactive) proactive[unit] = (uint8_t)pr;
            }
        }
        const int NW = (N + 31) / 32;
        for (int l = 0; l < L; l++) {
            uint32_t *bits = cache_bits + ((size_t)b * L + l) * NW;
            memset(bits, 0, sizeof(uint32_t) * (size_t)NW);
            for (int e = 0; e < N; e++)
                if (in_cache[(size_t)l * N + e]) bits[e / 32] |= 1u << (e % 32);
            if (aux_out) memcpy(aux_out + ((size_t)b * L + l) * N, aux + (size_t)l * N, 4 * (size_t)N);
            if (val_out) memcpy(val_out + ((size_t)b * L + l) * N, val + (size_t)l * N, 4 * (size_t)N);
        }
    }
    free(in_cache);
    free(count);
    free(aux);
    free(val);
    return rc;
}

/* ------------------------------------------------------------------------ */
/* soft Top-B cache-coverage losses (Sec. 3.1, 3.2, 3.3)                    */
/* ------------------------------------------------------------------------ */
/*
 * For a priority s over N experts and a target distribution q:
 *   theta_B(s) = the B-th largest entry of s,
 *   m_e(s)     = sigmoid((s_e - theta_B(s)) / tau),
 *   l(s, q)    = sum_e q_e (1 - m_e(s)).
 * Temporal:        l^T_{t,l}  = l(s^T_{t,l}, p^R_{t+1,l}),  s^T = p^R + p^T,
 *                  valid for t < T - 1 (a next-token target exists);
 * Spatio-Temporal: l^ST_{t,l} = l(s^ST_{t,l}, p^R_{t,l}),
 *                  s^ST = (p^R_{t-1,l} + p^T_{t-1,l}) + p^S_{rho(t,l)},
 *                  valid for t >= 1 (a previous token and a predecessor exist).
 * L_T, L_ST are the means over the valid positions of the B_s streams.
 * Readings: the native distributions stay differentiable as targets too
 * (Sec. 3.4), so d l / d q_e = 1 - m_e reaches the target's p^R; the
 * subgradient of theta_B goes to the element at position B under the total
 * order (score descending, index ascending); the priorities are formed in
 * fp32 exactly as the GPU forms them (so both pick the same theta element),
 * everything after that in fp64.
 * Outputs: loss [B_s][T][L][2] (l^T, l^ST; 0 where invalid) and, if grad is
 * not NULL, the gradient of w_T L_T + w_ST L_ST with respect to the logits of
 * the three heads, [B_s][T][L][3][N] (through p = softmax(z)); if grad_p is not
 * NULL, the gradient with respect to the probabilities, same layout.
 */
static double coverage_loss(int N, int Btop, double tau, const float *s, const float *q,
                            double *g, double *gq)
{
    int ord[ORACLE_MAX_N];
    order_desc_f32(s, N, ord);
    const int estar = ord[Btop - 1];
    const double theta = (double)s[estar];
    double loss = 0.0, sum_dm = 0.0;
    for (int e = 0; e < N; e++) {
        const double m = 1.0 / (1.0 + exp(-((double)s[e] - theta) / tau));
        loss += (double)q[e] * (1.0 - m);
        gq[e] = 1.0 - m;                                            /* d l / d q_e          */
        const double dm = (double)q[e] * m * (1.0 - m) / tau;      /* q_e dm_e/dx_e / tau */
        g[e] = -dm;                                                 /* d l / d s_e via s_e  */
        sum_dm += dm;
    }
    g[estar] += sum_dm;                                             /* via theta = s_{e*}   */
    return loss;
}

int oracle_cache_loss(int Bs, int T, int L, int N, int Btop, double tau, double w_T, double w_ST,
                      const float *probs, float *loss_out, double *grad, double *grad_p)
{
    if (Bs < 1 || T < 1 || L < 1 || N < 1 || N > ORACLE_MAX_N || Btop < 1 || Btop > N ||
        !(tau > 0.0))
        return -1;
    const size_t row = (size_t)3 * N;
    const size_t units = (size_t)Bs * T * L;
    double *dp = (double *)calloc(units * row, sizeof(double));   /* d objective / d p */
    double g[ORACLE_MAX_N], gq[ORACLE_MAX_N];
    float sv[ORACLE_MAX_N];
    const double nT = (double)Bs * (T - 1) * L, nST = (double)Bs * (T - 1) * L;
    const double cT = nT > 0 ? w_T / nT : 0.0, cST = nST > 0 ? w_ST / nST : 0.0;
    for (int b = 0; b < Bs; b++)
        for (int t = 0; t < T; t++)
            for (int l = 0; l < L; l++) {
                const size_t u = ((size_t)b * T + t) * L + l;
                const float *p = probs + u * row;
                float *lo = loss_out + u * 2;
                lo[0] = lo[1] = 0.0f;
                if (t + 1 < T) {                                    /* l^T_{t,l} */
                    const size_t uq = u + (size_t)L;                /* (t+1, l) */
                    const float *q = probs + uq * row;              /* p^R_{t+1,l} */
                    for (int e = 0; e < N; e++) sv[e] = p[e] + p[N + e];
                    lo[0] = (float)coverage_loss(N, Btop, tau, sv, q, g, gq);
                    for (int e = 0; e < N; e++) {
                        dp[u * row + e] += cT * g[e];               /* p^R_{t,l} */
                        dp[u * row + N + e] += cT * g[e];           /* p^T_{t,l} */
                        dp[uq * row + e] += cT * gq[e];             /* target p^R_{t+1,l} */
                    }
                }
                if (t >= 1) {                                       /* l^ST_{t,l} */
                    const size_t up = u - (size_t)L;                /* (t-1, l) */
                    const size_t ur = l > 0 ? u - 1 : (((size_t)b * T + (t - 1)) * L + (L - 1));
                    const float *pp = probs + up * row, *pr = probs + ur * row;
                    for (int e = 0; e < N; e++) {
                        const float a = pp[e] + pp[N + e];
                        sv[e] = a + pr[2 * N + e];
                    }
                    lo[1] = (float)coverage_loss(N, Btop, tau, sv, p, g, gq);   /* q = p^R_{t,l} */
                    for (int e = 0; e < N; e++) {
                        dp[up * row + e] += cST * g[e];             /* p^R_{t-1,l} */
                        dp[up * row + N + e] += cST * g[e];         /* p^T_{t-1,l} */
                        dp[ur * row + 2 * N + e] += cST * g[e];     /* p^S_{rho(t,l)} */
                        dp[u * row + e] += cST * gq[e];             /* target p^R_{t,l} */
                    }
                }
            }
    if (grad_p) memcpy(grad_p, dp, units * row * sizeof(double));
    if (grad) {                                 /* through each head's softmax: dz = p (dp - <p, dp>) */
        for (size_t u = 0; u < units; u++)
            for (int h = 0; h < 3; h++) {
                const float *p = probs + u * row + (size_t)h * N;
                const double *d = dp + u * row + (size_t)h * N;
                double dot = 0.0;
                for (int e = 0; e < N; e++) dot += (double)p[e] * d[e];
                for (int e = 0; e < N; e++) grad[u * row + (size_t)h * N + e] = (double)p[e] * (d[e] - dot);
            }
    }
    free(dp);
    return 0;
}
