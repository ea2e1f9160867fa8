/*
 * Cache-scan body of the oracle, included twice by crc_oracle.c with
 * REAL = double (SFX f64) and REAL = float (SFX f32).  TEST INFRASTRUCTURE.
 *
 * Each function follows the paper's Algorithm 2 (full inference step at
 * (t,l)) and Algorithm 1 (UpdateCache) literally: explicit sets, the loops in
 * the printed order, the argmin recomputed over the current set at each
 * iteration.  No closed form and no early exit is used here.
 */
#define CAT2_(a, b) a##_##b
#define CAT_(a, b) CAT2_(a, b)
#define FN(name) CAT_(name, SFX)

/* Positions of all N experts under the total order (score descending, index
 * ascending): insertion sort, an element only passes strictly smaller ones. */
static void FN(order_desc)(const REAL *s, int N, int *ord)
{
    for (int e = 0; e < N; e++) {
        int j = e;
        while (j > 0 && s[ord[j - 1]] < s[e]) {
            ord[j] = ord[j - 1];
            j--;
        }
        ord[j] = e;
    }
}

/* argmin over the members of a set: the LAST member under the total order,
 * i.e. the smallest score and, among equal scores, the highest index.  *gap
 * receives the relative gap to the next-smallest member (INFINITY if none). */
static int FN(argmin_last)(const REAL *s, const uint8_t *member, int N, double *gap)
{
    int v = -1;
    for (int e = 0; e < N; e++)
        if (member[e] && (v < 0 || s[e] <= s[v])) v = e;
    double g = INFINITY;
    if (v >= 0) {
        int has2 = 0;
        REAL m2 = 0;
        for (int e = 0; e < N; e++)
            if (member[e] && e != v && (!has2 || s[e] < m2)) {
                m2 = s[e];
                has2 = 1;
            }
        if (has2) g = rel_gap((double)s[v], (double)m2);
    }
    if (gap) *gap = g;
    return v;
}

/*
 * Algorithm 2, the refinement loop: pre-access refinement of a cache with priorities
 * sST (s^ST_{t,l}).  A = Top_R(sST) over all N experts; each candidate, in
 * descending order, is skipped when resident, inserted when the cache has a
 * free slot, else replaces the lowest resident only when strictly higher.
 * Each insertion is one proactive load; returns their number.  *margin is
 * lowered to the smallest relative gap met at any decision.
 */
int FN(oracle_refine)(int N, int C, int R, const REAL *sST, uint8_t *in_cache,
                      int *count, double *margin)
{
    int ord[ORACLE_MAX_N];
    double g, mg = margin ? *margin : INFINITY;
    int proactive = 0;
    FN(order_desc)(sST, N, ord);
    int nA = R < N ? R : N;                 /* A = Top_R(s^ST)                 */
    for (int i = 0; i + 1 < N && i < nA; i++) {
        g = rel_gap((double)sST[ord[i]], (double)sST[ord[i + 1]]);
        if (g < mg) mg = g;
    }
    for (int i = 0; i < nA; i++) {          /* descending order of s^ST        */
        int e = ord[i];
        if (in_cache[e]) continue;
        if (*count < C) {                   /* proactive load into a free slot */
            in_cache[e] = 1;
            (*count)++;
            proactive++;
        } else {
            int v = FN(argmin_last)(sST, in_cache, N, &g);
            if (g < mg) mg = g;
            g = rel_gap((double)sST[e], (double)sST[v]);
            if (g < mg) mg = g;
            if (sST[e] > sST[v]) {          /* strictly higher: replace lowest */
                in_cache[v] = 0;
                in_cache[e] = 1;
                proactive++;
            }
        }
    }
    if (margin) *margin = mg;
    return proactive;
}

/*
 * Algorithm 1, UpdateCache(C, S, s, C): D = S \ C+ walked in ascending
 * index; a free slot takes e directly, otherwise the lowest-priority
 * non-selected resident v = argmin_{V = C+ \ S} s is evicted for e.
 * inS[N] marks S.  Returns |D| (the demand-loaded experts).
 */
int FN(oracle_update_cache)(int N, int C, const REAL *s, const uint8_t *inS,
                            uint8_t *in_cache, int *count, double *margin)
{
    uint8_t inD[ORACLE_MAX_N], inV[ORACLE_MAX_N];
    double g, mg = margin ? *margin : INFINITY;
    int nD = 0;
    for (int e = 0; e < N; e++) {           /* D = S \ C+ */
        inD[e] = (uint8_t)(inS[e] && !in_cache[e]);
        nD += inD[e];
    }
    for (int e = 0; e < N; e++) {
        if (!inD[e]) continue;
        if (*count < C) {
            in_cache[e] = 1;
            (*count)++;
        } else {
            for (int u = 0; u < N; u++) inV[u] = (uint8_t)(in_cache[u] && !inS[u]);
            int v = FN(argmin_last)(s, inV, N, &g);   /* V = C+ \ S */
            if (g < mg) mg = g;
            in_cache[v] = 0;
            in_cache[e] = 1;
        }
    }
    if (margin) *margin = mg;
    return nD;
}

/*
 * One access at (t,l) for one chain (Algorithm 2).  State: in_cache[N] (0/1),
 * *count = |C|, aT[N] = s^T of the previous token at this layer (ignored when
 * t == 0).  pS_pred = p^S of the causal predecessor rho(t,l); read only when
 * R > 0 and t >= 1.  Outputs: topk_out[K] in rank order, demand misses,
 * proactive loads, and the smallest relative gap met at any decision of this
 * access (the unit's decision margin).  Returns 0, or -1 on invalid sizes.
 */
int FN(oracle_step)(int N, int K, int C, int R, int t,
                    const REAL *pR, const REAL *pT, const REAL *pS_pred,
                    uint8_t *in_cache, int *count, REAL *aT,
                    int *topk_out, int *misses_out, int *proactive_out,
                    double *margin_out)
{
    if (N < 1 || N > ORACLE_MAX_N || K < 1 || K > N || C < K || C > N || R < 0)
        return -1;
    int ord[ORACLE_MAX_N];
    REAL sT[ORACLE_MAX_N], sST[ORACLE_MAX_N];
    double margin = INFINITY, g;
    int proactive = 0;

    /* Algorithm 2, refinement: pre-access refinement (full mode, t >= 1) */
    if (R > 0 && t >= 1) {
        for (int e = 0; e < N; e++) {
            REAL a = aT[e];                 /* a^T = p^R_{t-1,l} + p^T_{t-1,l} */
            sST[e] = a + pS_pred[e];        /* s^ST = a^T + p^S_{rho(t,l)}     */
        }
        proactive = FN(oracle_refine)(N, C, R, sST, in_cache, count, &margin);
    }

    /* Algorithm 2, access: native Top-K on p^R (the set boundary K/K+1 is the decision;
     * the order inside the set only orders the trace) */
    FN(order_desc)(pR, N, ord);
    uint8_t inS[ORACLE_MAX_N];
    memset(inS, 0, (size_t)N);
    for (int k = 0; k < K; k++) {
        topk_out[k] = ord[k];
        inS[ord[k]] = 1;
    }
    if (K < N) {
        g = rel_gap((double)pR[ord[K - 1]], (double)pR[ord[K]]);
        if (g < margin) margin = g;
    }

    /* Algorithm 2, retention score: s^T = p^R + p^T */
    for (int e = 0; e < N; e++) sT[e] = pR[e] + pT[e];

    /* Algorithm 2, demand load of S \ C~, then UpdateCache (Algorithm 1) */
    int misses = FN(oracle_update_cache)(N, C, sT, inS, in_cache, count, &margin);
    for (int e = 0; e < N; e++) aT[e] = sT[e];

    *misses_out = misses;
    *proactive_out = proactive;
    if (margin_out) *margin_out = margin;
    return 0;
}

typedef struct {
    int B, T, L, N, K, C, R;
    const REAL *probs;
    uint8_t *topk, *misses, *proactive;
    double *margins;
    uint32_t *cache_bits;
    REAL *aT_out;
    uint64_t *counters;
    int b_begin, b_end;
    int status;
    int ties_exempt;
} FN(scan_job);

static void *FN(scan_worker)(void *arg)
{
    FN(scan_job) *j = (FN(scan_job) *)arg;
    const int L = j->L, N = j->N, K = j->K, T = j->T;
    const size_t row = (size_t)3 * N;
    uint8_t *in_cache = (uint8_t *)calloc((size_t)L * N, 1);
    int *count = (int *)calloc((size_t)L, sizeof(int));
    REAL *aT = (REAL *)calloc((size_t)L * N, sizeof(REAL));
    int topk[ORACLE_MAX_N];
    j->status = 0;
    exact_ties_exempt = j->ties_exempt;
    for (int b = j->b_begin; b < j->b_end; b++) {
        memset(in_cache, 0, (size_t)L * N);
        memset(count, 0, sizeof(int) * (size_t)L);
        memset(aT, 0, sizeof(REAL) * (size_t)L * N);
        uint64_t *ctr = j->counters + (size_t)b * L * 3;
        memset(ctr, 0, sizeof(uint64_t) * (size_t)L * 3);
        for (int t = 0; t < T; t++) {
            for (int l = 0; l < L; l++) {
                size_t unit = ((size_t)b * T + t) * L + l;
                const REAL *pR = j->probs + unit * row;
                const REAL *pT = pR + N;
                const REAL *pS = NULL;              /* p^S_{rho(t,l)} */
                if (l > 0)
                    pS = j->probs + (unit - 1) * row + 2 * N;
                else if (t > 0)
                    pS = j->probs + (((size_t)b * T + (t - 1)) * L + (L - 1)) * row + 2 * N;
                int mi, pr;
                double mg;
                if (FN(oracle_step)(N, K, j->C, j->R, t, pR, pT, pS,
                                    in_cache + (size_t)l * N, &count[l], aT + (size_t)l * N,
                                    topk, &mi, &pr, &mg) != 0) {
                    j->status = -1;
                    goto done;
                }
                ctr[l * 3 + 0] += (uint64_t)(K - mi);
                ctr[l * 3 + 1] += (uint64_t)mi;
                ctr[l * 3 + 2] += (uint64_t)pr;
                if (j->topk)
                    for (int k = 0; k < K; k++) j->topk[unit * K + k] = (uint8_t)topk[k];
                if (j->misses) j->misses[unit] = (uint8_t)mi;
                if (j->proactive) j->proactive[unit] = (uint8_t)pr;
                if (j->margins) j->margins[unit] = mg;
            }
        }
        const int NW = (N + 31) / 32;
        for (int l = 0; l < L; l++) {
            uint32_t *bits = j->cache_bits + ((size_t)b * L + l) * NW;
            memset(bits, 0, sizeof(uint32_t) * (size_t)NW);
            for (int e = 0; e < N; e++)
                if (in_cache[(size_t)l * N + e]) bits[e / 32] |= 1u << (e % 32);
            if (j->aT_out)
                memcpy(j->aT_out + ((size_t)b * L + l) * N, aT + (size_t)l * N,
                       sizeof(REAL) * (size_t)N);
        }
    }
done:
    exact_ties_exempt = 0;
    free(in_cache);
    free(count);
    free(aT);
    return NULL;
}

/*
 * Whole scan over B independent streams, T tokens, L layers, cold start.
 * probs [B][T][L][3][N] (the S head is read only when R > 0).
 * Outputs (any trace pointer may be NULL): topk [B][T][L][K] in rank order,
 * misses / proactive [B][T][L], margins [B][T][L], cache_bits [B][L][ceil(N/32)],
 * aT_out [B][L][N] (s^T of the last token), counters [B][L][3] = hits,
 * demand misses, proactive loads.  ties_exempt: gaps of exactly zero do not
 * lower the margins (ties built on purpose).  Returns 0 or -1.
 */
int FN(oracle_scan)(int B, int T, int L, int N, int K, int C, int R,
                    const REAL *probs, uint8_t *topk, uint8_t *misses,
                    uint8_t *proactive, double *margins, uint32_t *cache_bits,
                    REAL *aT_out, uint64_t *counters, int nthreads, int ties_exempt)
{
    if (B < 0 || T < 0 || L < 1 || N < 1 || N > ORACLE_MAX_N || K < 1 || K > N ||
        C < K || C > N || R < 0)
        return -1;
    if (nthreads < 1) nthreads = 1;
    if (nthreads > B) nthreads = B > 0 ? B : 1;
    if (nthreads > 256) nthreads = 256;
    FN(scan_job) jobs[256];
    pthread_t th[256];
    int per = (B + nthreads - 1) / nthreads;
    for (int k = 0; k < nthreads; k++) {
        FN(scan_job) jj = {B, T, L, N, K, C, R, probs, topk, misses, proactive,
                           margins, cache_bits, aT_out, counters,
                           k * per, (k + 1) * per < B ? (k + 1) * per : B, 0, ties_exempt};
        jobs[k] = jj;
    }
    if (nthreads == 1) {
        FN(scan_worker)(&jobs[0]);
    } else {
        for (int k = 0; k < nthreads; k++) pthread_create(&th[k], NULL, FN(scan_worker), &jobs[k]);
        for (int k = 0; k < nthreads; k++) pthread_join(th[k], NULL);
    }
    for (int k = 0; k < nthreads; k++)
        if (jobs[k].status) return -1;
    return 0;
}

#undef FN
#undef CAT_
#undef CAT2_
