/*
 * crc.h -- C ABI of the GB300 (sm_103a) cache-aware MoE routing library.
 *
 * For a batch of B independent decode streams, T tokens and L MoE layers
 * with N routed experts each, the library computes the per-token, per-layer
 * routing and expert-residency step of cache-aware MoE decoding ("Cache-Aware
 * Joint Router Adaptation for Memory-Efficient MoE Inference"):
 *
 *   p^R = softmax(W^R_l h), S = TopK(p^R)               (Sec. 2)
 *   p^T = softmax(W^T_l h), s^T = p^R + p^T             (Sec. 3.2)
 *   p^S = softmax(W^S_l h), s^ST = s^T_{t-1} + p^S_rho  (Sec. 3.3)
 *   pre-access refinement (Algorithm 2, R > 0), access, post-access
 *   retention UpdateCache (Algorithm 1) on a C-slot cache per (stream, layer),
 *   counting accesses, demand misses and proactive loads (Sec. 4.1 Metrics).
 *
 * Notation: the paper's cache capacity B is called C here; B here is the
 * number of independent decode streams.  Layers and tokens are 0-indexed,
 * so the causal predecessor is rho(t,0) = (t-1, L-1), rho(t,l) = (t, l-1).
 *
 * Conventions for every entry point:
 *  - Pointers named *_dev are device pointers the caller allocated (the
 *    library allocates no device memory except where stated); *_host are
 *    host pointers.  bf16 data is passed as uint16_t bit patterns.
 *  - `stream` is a cudaStream_t (NULL = legacy default stream).  Calls are
 *    asynchronous on it unless stated; they return after enqueueing.
 *  - Return value: CRC_OK (0) or an error code below.  Argument errors are
 *    detected on the host before anything is enqueued.  Errors found on the
 *    device (a bounded wait that ran out, a state mismatch) are latched in
 *    the state's error word and reported by crc_state_read(), or, for calls
 *    without a state, by crc_device_error().  Nothing aborts or prints.
 *  - Policy decisions use one total order: score descending, then expert
 *    index ascending.  Top-K / Top-R take its first elements; every argmin
 *    takes its last (smallest score, ties to the highest index).  The
 *    refinement test is strict.  No refinement at a stream's first token.
 *    Caches start empty.  Scores are probabilities (finite, >= 0).
 *  - Limits: 16 <= N <= 128 with N % 16 == 0 for the router entry points
 *    (N <= 256 for crc_cache_scan); 1 <= K <= min(C, 32); K <= C <= N;
 *    0 <= R <= N; d % 8 == 0; L >= 1; B >= 1.
 */
#ifndef CRC_H
#define CRC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

enum {
    CRC_OK = 0,
    CRC_EINVAL = 1,        /* null / misaligned pointer, bad size, T < 0      */
    CRC_EUNSUPPORTED = 2,  /* sizes outside the limits above                  */
    CRC_ECUDA = 3,         /* a CUDA runtime call or launch failed            */
    CRC_ETIMEOUT = 4,      /* a bounded device wait ran out (latched)         */
    CRC_ESTATE = 5,        /* state buffer too small, uninitialised or made
                              for another problem (latched when seen on GPU)  */
    CRC_EDEVICE = 6,       /* other device-side failure (latched)             */
    CRC_ENOMEM = 7         /* host memory could not be mapped                 */
};

/* The problem statement (Sec. 2): sizes and budgets.  One per state. */
typedef struct crc_problem {
    int32_t L;              /* MoE layers                                     */
    int32_t N;              /* routed experts per layer                       */
    int32_t K;              /* native Top-K                                   */
    int32_t d;              /* hidden size                                    */
    int32_t C;              /* cache slots per layer (the paper's B)          */
    int32_t R;              /* refinement budget; 0 = update-only mode        */
    int32_t B;              /* independent decode streams                     */
    int32_t reserved;       /* must be 0                                      */
    uint64_t expert_bytes;  /* bytes of one expert transfer (S_exp)           */
} crc_problem;

/* Optional per-access trace of one call, device pointers, each may be NULL.
 * T is the call's token count and t the token index within the call.  The
 * sets are bitmasks of NW = ceil(N / 32) words per access (expert e is bit
 * e % 32 of word e / 32); the cache sets and the Top-K set are written by the
 * method's scan only (crc_cache_scan, crc_route_and_cache), not by the
 * comparison policies.  The native Top-K comes in two forms: topk_dev in rank
 * order (p^R descending, ties to the lower index), and topk_set_dev, the same
 * experts as a set, which is all that the cache decisions use (Sec. 2:
 * S = TopK(p^R) is a set).  crc_route_and_cache runs as one fused kernel
 * with any trace that does not ask for topk_dev (see there). */
typedef struct crc_trace {
    uint8_t *topk_dev;       /* [B][T][L][K] native Top-K, rank order          */
    uint8_t *misses_dev;     /* [B][T][L] demand misses |S \ C~|               */
    uint8_t *proactive_dev;  /* [B][T][L] proactive loads of the refinement    */
    uint32_t *cache_mid_dev; /* [B][T][L][NW] cache after Algorithm 2 (C~)     */
    uint32_t *cache_after_dev; /* [B][T][L][NW] cache after UpdateCache      */
    uint32_t *topk_set_dev;  /* [B][T][L][NW] native Top-K S as a set          */
} crc_trace;

/* Totals over all streams and layers since crc_state_init (Sec. 4.1). */
typedef struct crc_stats {
    uint64_t accesses;       /* A = L * K * tokens * B                         */
    uint64_t hits;           /* A - D                                          */
    uint64_t misses;         /* D, demand misses                               */
    uint64_t proactive;      /* P, proactive loads                             */
    uint64_t traffic_bytes;  /* (D + P) * expert_bytes                         */
    uint64_t tokens;         /* tokens processed per stream                    */
    uint32_t error;          /* latched device error code, CRC_OK if none      */
    uint32_t reserved;
} crc_stats;

/* ------------------------------------------------------------------------ */
/* State: a caller-owned device buffer holding, per (stream, layer), the    */
/* cache set C_{t,l} that Algorithms 1 and 2 update (bitmask), the carried  */
/* retention score s^T_{t-1,l} (= a^T_{t,l} of Sec. 3.3, fp32 [N]) and the  */
/* hit / miss / proactive counters of Sec. 4.1; per stream the carried      */
/* Spatio prediction p^S_{t-1,L-1} (the wrap-around causal predecessor of   */
/* layer 0, Sec. 3.3); and the next token index.  Successive calls on one   */
/* state continue the same streams: processing T tokens in chunks gives     */
/* bit-identical results to one call.  Two calls on one state must not run  */
/* concurrently.                                                            */
/* ------------------------------------------------------------------------ */

/* Bytes needed for the state of problem p (0 if p is invalid). */
size_t crc_state_bytes(const crc_problem *p);

/* Cold start: empty caches (the not-full branches of Algorithms 1 and 2
 * fill them), zero counters, token 0.  state_dev must be 256-byte aligned and
 * hold crc_state_bytes(p) bytes.  Asynchronous. */
int crc_state_init(const crc_problem *p, void *state_dev, size_t state_bytes, void *stream);

/* Synchronises `stream`, then reads the state back: the Sec. 4.1 totals
 * into *out (required); optionally cache bitmasks [B][L][ceil(N/32)] (bit e % 32 of
 * word e / 32 set when expert e is resident), the carried retention scores
 * [B][L][N] and per-(stream, layer) counters [B][L][3] = hits, misses,
 * proactive.  Returns the latched device error if there is one. */
int crc_state_read(const crc_problem *p, const void *state_dev, size_t state_bytes,
                   crc_stats *out, uint32_t *cache_bits_host, float *retention_host,
                   uint64_t *chain_counters_host, void *stream);

/* The paper's reported metrics (Sec. 4.1 Metrics) from the totals of
 * crc_state_read, over all B streams: with A accesses, D demand misses, P
 * proactive loads, S_exp = expert_bytes and B * tokens decode tokens,
 *   hit                  = 1 - D / A             (NaN when A = 0)
 *   adj_hit              = (A - D) / (A + P)     (NaN when A + P = 0)
 *   traffic_bytes        = (D + P) * S_exp
 *   load_per_token_bytes = (D + P) * S_exp / (B * tokens)   (0 with no token)
 * Host-only arithmetic; CRC_EINVAL for a null pointer or invalid problem. */
typedef struct crc_report {
    double hit;
    double adj_hit;
    double traffic_bytes;
    double load_per_token_bytes;
} crc_report;
int crc_metrics(const crc_problem *p, const crc_stats *s, crc_report *out);

/* Exposed expert-loading cost per decode token under the overlap model of
 * the paper's appendix on asynchronous transfer overlap: each expert
 * transfer takes c_exp seconds, demand transfers are fully exposed and a
 * fraction eta of the proactive ones is hidden behind computation,
 *   *t_load = c_exp / (B * tokens) * (D + (1 - eta) * P)   (0 with no token).
 * Host-only; CRC_EINVAL for a null pointer, an invalid problem, eta outside
 * [0, 1] or a negative or non-finite c_exp. */
int crc_load_time(const crc_problem *p, const crc_stats *s, double c_exp, double eta,
                  double *t_load);

/* ------------------------------------------------------------------------ */
/* Hot path                                                                 */
/* ------------------------------------------------------------------------ */

/* Router heads (Sec. 2, 3.2, 3.3): for every unit (b, t, l),
 *   scores[b][t][l][x][:] = softmax(W_cat[l][x*N:(x+1)*N] . hidden[b][t][l]),
 * x = 0 (native R), 1 (Temporal T), 2 (Spatio S); heads = 2 skips S (the
 * S slot of `scores` is then left untouched).  One bf16 GEMM per layer on
 * the tensor cores with fp32 accumulation, softmax in fp32.
 *   hidden_dev  bf16 [B][T][L][d], 16-byte aligned
 *   w_cat_dev   bf16 [L][3N][d], heads ordered R, T, S, 16-byte aligned
 *   scores_dev  fp32 [B][T][L][3][N], 16-byte aligned
 * T = 0 is a no-op.  Device-side failures: crc_device_error(). */
int crc_route_scores(const crc_problem *p, const uint16_t *hidden_dev,
                     const uint16_t *w_cat_dev, int32_t T, int32_t heads,
                     float *scores_dev, void *stream);

/* Cache simulation over T tokens (Algorithm 2 with Algorithm 1, Sec. 4.1
 * accounting) from router probabilities, one warp per (stream, layer):
 *   scores_dev  fp32 [B][T][L][3][N] as written by crc_route_scores (the S
 *               head is read only when R > 0), 16-byte aligned.
 * Continues the streams held in `state_dev`; `trace` may be NULL. */
int crc_cache_scan(const crc_problem *p, const float *scores_dev, int32_t T,
                   void *state_dev, size_t state_bytes, const crc_trace *trace,
                   void *stream);

/* Comparison policies of the paper's evaluation (Sec. 4: the cache-update
 * baselines LRU, LFU and LRFU with lambda = 0.5; Sec. 4.3 and the ablation
 * appendix: Spatio-only, i.e. Algorithm 2's refinement on
 * s^S = p^R_{t-1} + p^S_rho with LRU eviction for demand misses). */
enum { CRC_POLICY_LRU = 1, CRC_POLICY_LFU = 2, CRC_POLICY_LRFU = 3, CRC_POLICY_SPATIO_LRU = 4 };

/* The cache simulation of crc_cache_scan under a comparison policy, same
 * arguments plus:
 *   policy         one of CRC_POLICY_*; a state belongs to the policy of its
 *                  first call (a later call with another policy, or a call of
 *                  crc_cache_scan / crc_route_and_cache on it, latches
 *                  CRC_ESTATE);
 *   lambda_halves  LRFU's lambda in halves (0..8; 1 = the paper's 0.5),
 *                  ignored by the other policies.
 * LRU, LFU and LRFU demand-load S \ C and, with the cache full, evict the
 * resident outside S with the lowest priority (token of last use; accesses
 * since insertion; CRF * 2^(-lambda (t - t_last)) with the CRF updated to
 * 1 + 2^(-lambda (t - t_last)) CRF at each use), ties to the highest expert
 * index; they make no proactive load.  R is used by Spatio-only only.
 * CRC_EINVAL for a policy or lambda outside these ranges. */
int crc_cache_scan_policy(const crc_problem *p, const float *scores_dev, int32_t T,
                          void *state_dev, size_t state_bytes, const crc_trace *trace,
                          int32_t policy, int32_t lambda_halves, void *stream);

/* Synchronises `stream` and copies a comparison policy's integer priorities
 * [B][L][N] (LRU, Spatio-only, LRFU: token of last use; LFU: accesses since
 * insertion) into aux_host; its float priorities (LRFU: CRF; Spatio-only:
 * p^R of the last token) come with crc_state_read's retention array. */
int crc_state_read_aux(const crc_problem *p, const void *state_dev, size_t state_bytes,
                       uint32_t *aux_host, void *stream);

/* Bytes of workspace crc_route_and_cache uses to process `chunk_tokens`
 * tokens per pass (the router scores of one chunk). */
size_t crc_workspace_bytes(const crc_problem *p, int32_t chunk_tokens);

/* Workspace bytes with which crc_route_and_cache runs as ONE fused kernel
 * (router heads on the tensor cores and the scan together; the router scores
 * then only pass through a ring of tiles in the workspace).  The fused kernel
 * serves calls with K <= 8 and 16 <= N <= 128 whose trace, if any, does not
 * ask for the Top-K in rank order (crc_trace.topk_dev); other calls, or
 * smaller workspaces, take the chunked two-kernel path.  0 if p is invalid. */
size_t crc_fused_workspace_bytes(const crc_problem *p);

/* The whole step of the paper's decoding loop over T tokens: the router
 * heads (Sec. 2, 3.2, 3.3), then per access the pre-access refinement and
 * access of Algorithm 2 with UpdateCache (Algorithm 1) and the Sec. 4.1
 * accounting -- the same results as crc_route_scores followed by
 * crc_cache_scan (bit for bit).
 * hidden_dev bf16 [B][T][L][d]; w_cat_dev bf16 [L][3N][d] (the S head is
 * not computed when R = 0).  The router scores never leave the workspace.
 * With workspace_bytes >= crc_fused_workspace_bytes(p), K <= 8 and a trace
 * that leaves topk_dev NULL (or no trace) the call is one fused kernel; for N = 128 with 128-token tiles of one stream
 * (T > 64) and an even stream count its GEMM runs on CTA pairs (clusters of
 * two, tcgen05 cta_group::2), otherwise one CTA per tile, with the same
 * results.  The pair kernel is a cooperative cluster launch; with the
 * environment variable CRC_PLAIN_CLUSTER_LAUNCH=1 (read once per process) it
 * is launched without the cooperative attribute, for kernel profilers that
 * cannot replay cooperative cluster launches (same kernel, same grid, which
 * fits the GPU at once; a stall would end in CRC_ETIMEOUT).  Without that workspace, workspace_dev holds the scores of one
 * chunk of tokens, the chunk length being the largest that fits (at least one
 * token must fit, see crc_workspace_bytes).  256-byte alignment for the
 * workspace. */
int crc_route_and_cache(const crc_problem *p, const uint16_t *hidden_dev,
                        const uint16_t *w_cat_dev, int32_t T, void *state_dev,
                        size_t state_bytes, const crc_trace *trace,
                        void *workspace_dev, size_t workspace_bytes, void *stream);

/* Device bytes of the two staging halves crc_route_and_cache_host uses for
 * chunks of `chunk_tokens` tokens: 2 x B x chunk_tokens x L x d bf16, each
 * half rounded up to 256 bytes.  0 if p is invalid or chunk_tokens < 1. */
size_t crc_host_staging_bytes(const crc_problem *p, int32_t chunk_tokens);

/* Pinned (page-locked, CUDA-registered) host memory for the host-input call:
 * an anonymous mapping aligned to the kernel's transparent huge-page size,
 * advised MADV_HUGEPAGE and faulted in before registration, so that a
 * multi-GB buffer is covered by few large pages (copies of a 12.9 GB buffer
 * in cudaHostAlloc's small pages ran at 40-60 GB/s about one time in three,
 * against a steady 210 GB/s from huge pages).  *out receives the pointer
 * (huge-page aligned, at least `bytes` long); CRC_ENOMEM if the mapping fails,
 * CRC_ECUDA if registration fails (nothing is left allocated).  Free with
 * crc_host_free only; crc_host_free(NULL) is a no-op and a pointer this
 * library did not hand out gives CRC_EINVAL. */
int crc_host_alloc(size_t bytes, void **out);
int crc_host_free(void *ptr);

/* crc_route_and_cache with the hidden states in HOST memory (no counterpart
 * in the paper: the copy from the host is the serving system's, Sec. 2).
 *   hidden_host   bf16 [B][T][L][d] in host memory, 16-byte aligned; pinned
 *                 (page-locked, e.g. from crc_host_alloc) memory lets the
 *                 copies overlap the compute; pageable memory gives the same
 *                 results without overlap
 *   chunk_tokens  tokens per copy; the call moves tokens [t0, t0 + chunk) of
 *                 every stream into one staging half (a 2-D copy on a copy
 *                 stream the call creates and destroys) while `stream` runs
 *                 the step on the previous chunk in the other half
 *   staging_dev   device buffer of crc_host_staging_bytes(p, min(chunk, T))
 *                 bytes, 256-byte aligned
 * workspace_dev / workspace_bytes as in crc_route_and_cache (with
 * crc_fused_workspace_bytes every chunk is one fused kernel); no trace.
 * Results are bit-identical to crc_route_and_cache over all T tokens (the
 * calls on successive chunks continue the same state).  The call returns
 * once everything is queued; all of its work, copies included, is ordered
 * before later work on `stream`, so neither the host buffer nor the staging
 * buffer may be reused before `stream` has passed the call.  On an error
 * part of the work may have been queued: synchronise `stream` before
 * freeing the buffers. */
int crc_route_and_cache_host(const crc_problem *p, const uint16_t *hidden_host,
                             const uint16_t *w_cat_dev, int32_t T, int32_t chunk_tokens,
                             void *state_dev, size_t state_bytes, void *staging_dev,
                             size_t staging_bytes, void *workspace_dev, size_t workspace_bytes,
                             void *stream);

/* Failure-path probe (no counterpart in the paper).  Launches one warp that
 * waits on something that never happens -- kind 0: a flag nothing sets,
 * through the bounded flag wait of the fused kernel; kind 1: an mbarrier
 * phase nothing completes, through the bounded mbarrier wait of every
 * tcgen05 kernel -- for limit_ns nanoseconds (clamped to [1 ms, 2 s], the
 * hot-path limit being 2 s).  The expired wait latches CRC_ETIMEOUT in the
 * state's error word, as a stalled hot-path kernel would, and the kernel
 * returns: nothing traps or faults and the context stays usable.
 * crc_state_read then reports CRC_ETIMEOUT.  state_dev: an initialised state
 * of p (256-byte aligned).  Uses a two-word array compiled into the library:
 * do not run two probes at once.  CRC_EINVAL for another kind. */
int crc_wait_probe(const crc_problem *p, void *state_dev, size_t state_bytes, int32_t kind,
                   uint64_t limit_ns, void *stream);

/* ------------------------------------------------------------------------ */
/* Allocation-free variant (no counterpart in the paper)                    */
/* ------------------------------------------------------------------------ */

/* Capacity of the library's built-in scratch array, per GPU. */
#define CRC_NOALLOC_SCRATCH_BYTES ((size_t)32 << 20)

/* crc_route_and_cache without a workspace argument, for callers that cannot
 * allocate device memory when they call in: for example code running inside a
 * serving framework that reserved all device memory for its own pool at
 * start-up, or a plug-in whose host application forbids allocation after
 * initialisation (cudaMalloc / cudaFree may also synchronise the whole
 * device, which a latency-bound decode loop cannot afford).  The caller still
 * provides every input and output (hidden states, weights, state, trace).
 * This call allocates nothing: its scratch is a fixed array compiled into the
 * library, CRC_NOALLOC_SCRATCH_BYTES bytes on every GPU where the library is
 * loaded, kept until the process exits.  The array takes one of two layouts,
 * exactly as a caller workspace of that size would in crc_route_and_cache:
 *  - when crc_fused_workspace_bytes(p) <= CRC_NOALLOC_SCRATCH_BYTES (small
 *    problems: few streams and layers) and the trace, if any, leaves topk_dev
 *    NULL, the call is the fused kernel, with its control words and its ring
 *    of router-score tiles in the array (the control words are cleared by the
 *    call itself before the kernel starts);
 *  - otherwise the router scores of each chunk of tokens go to the array, the
 *    chunk being the largest number of tokens whose scores (B * L * 3N * 4
 *    bytes per token) fit in it; a problem whose scores for one token do not
 *    fit is refused with CRC_EUNSUPPORTED before anything is enqueued.
 * The first call on a device looks up that device's copy of the array (once
 * per device, with the device current); make that first call before any
 * stream capture.  The address is kept for the life of the process, so a
 * device reset (cudaDeviceReset) after that first call is not supported.
 * All calls share the one array per device and it keeps the last call's
 * contents (nothing in it needs to start at zero beyond what each call
 * clears itself), so calls whose kernels may overlap on the GPU -- unordered
 * streams or concurrent host threads -- race on it: order them.  Results are
 * bit-identical to crc_route_and_cache. */
int crc_route_and_cache_noalloc(const crc_problem *p, const uint16_t *hidden_dev,
                                const uint16_t *w_cat_dev, int32_t T, void *state_dev,
                                size_t state_bytes, const crc_trace *trace, void *stream);

/* ------------------------------------------------------------------------ */
/* Support                                                                  */
/* ------------------------------------------------------------------------ */

/* Soft Top-B cache-coverage losses and their gradient (Sec. 3.1-3.4): the
 * training objective of the Temporal and Spatio heads, over whole sequences
 * (tokens 0 .. T-1 of every stream).  With theta_B(s) the top_b-th largest
 * entry of s, m_e(s) = sigmoid((s_e - theta_B(s)) / tau) and
 * l(s, q) = sum_e q_e (1 - m_e(s)):
 *   l^T_{t,l}  = l(p^R_{t,l} + p^T_{t,l}, p^R_{t+1,l})                  t < T-1
 *   l^ST_{t,l} = l(p^R_{t-1,l} + p^T_{t-1,l} + p^S_{rho(t,l)}, p^R_{t,l}) t >= 1
 *   L_T, L_ST  = their means over the B (T-1) L valid positions each.
 * The priorities are summed in fp32 in that order (as the cache scan sums
 * them), theta_B is exact on those fp32 values and its subgradient goes to
 * the element at position top_b of the total order; the rest is fp32, the
 * means are fp64 sums in a fixed order (no atomics: results are
 * deterministic).
 *   probs_dev   fp32 [B][T][L][3][N] (crc_route_scores' layout; finite,
 *               >= 0), 16-byte aligned.  heads = 2 reads the R and T heads
 *               only and computes l^T alone (l^ST = L_ST = 0, the S rows of
 *               grad_dev untouched).
 *   top_b       1..N;  tau > 0;  w_T, w_ST finite (the objective is
 *               w_T L_T + w_ST L_ST).
 *   loss_dev    fp32 [B][T][L][2]: l^T, l^ST per position (0 where not
 *               valid), or NULL.
 *   means_dev   fp64 [2] = (L_T, L_ST), or NULL.  Needs workspace_dev with
 *               crc_loss_workspace_bytes(p, T) bytes, 256-byte aligned.
 *   grad_dev    fp32 [B][T][L][3][N], or NULL: the gradient of the objective
 *               with respect to each head's logits z (p = softmax(z)); the
 *               native distributions are differentiable both as priorities
 *               and as targets.  16-byte aligned, not aliasing probs_dev.
 * K, C and R of the problem are not used.  T = 0 is a no-op.  Device-side
 * failures: crc_device_error(). */
size_t crc_loss_workspace_bytes(const crc_problem *p, int32_t T);
int crc_cache_loss(const crc_problem *p, const float *probs_dev, int32_t T, int32_t heads,
                   int32_t top_b, double tau, double w_T, double w_ST, float *loss_dev,
                   double *means_dev, float *grad_dev, void *workspace_dev,
                   size_t workspace_bytes, void *stream);

/* Expert transfers (the expert pool of Sec. 2 and the transfers counted in
 * Sec. 4.1): the cache simulation's load decisions for one stream as copies
 * of expert weights from a host pool into a device cache of C slots per
 * layer.  One planned copy: */
typedef struct crc_transfer {
    int32_t t;          /* token of the access (index into the trace)          */
    int32_t l;          /* layer                                               */
    int32_t expert;     /* expert loaded                                       */
    int32_t slot;       /* destination slot, 0 .. C-1 of layer l               */
    int32_t evicted;    /* expert that left that slot in this phase, -1 if free */
    int32_t proactive;  /* 1: Algorithm 2 proactive load; 0: demand load       */
} crc_transfer;

/* Host-only planning from one stream's cache trace (crc_trace's cache_mid and
 * cache_after of that stream, host copies, [T][L][NW] each).  Per access, the
 * experts that entered the cache in the refinement phase (C~ \ C) are the
 * proactive loads and those that entered in UpdateCache (C+ \ C~) the demand
 * loads, so the plan holds exactly P + D copies; an expert that leaves frees
 * its slot.  Slots: within a phase the freed slots are taken first (ascending
 * slot), by the loaded experts in ascending expert order, then free slots.
 *   start_host   [L][NW] cache before token 0, checked against slot_expert
 *                (NULL: not checked);
 *   slot_expert  [L][C] in: the expert in each slot before token 0 (-1 free);
 *                out: after the last token;
 *   out          room for max_out copies, or NULL to count only;
 *                *n_out receives the number of copies.
 * CRC_EINVAL on bad sizes, inconsistent masks (more than C members, an
 * expert in two slots) or more copies than max_out (with out given). */
int crc_transfer_plan(const crc_problem *p, int32_t T, const uint32_t *mid_host,
                      const uint32_t *after_host, const uint32_t *start_host,
                      int32_t *slot_expert, crc_transfer *out, int64_t max_out,
                      int64_t *n_out);

/* Enqueues the planned copies on `stream`, in plan order, one
 * cudaMemcpyAsync of expert_bytes each: from pool_host (pinned host memory,
 * pool_experts expert images; copy (l, e) reads image (l * N + e) %
 * pool_experts, so a pool of L * N images holds every expert once) to
 * slots_dev [L][C][expert_bytes].  Asynchronous; CRC_ECUDA if a copy cannot
 * be enqueued. */
int crc_transfer_replay(const crc_problem *p, const crc_transfer *plan, int64_t n,
                        const void *pool_host, int64_t pool_experts, void *slots_dev,
                        void *stream);

/* Synchronises the device and returns (then clears) the error latched by
 * calls without a state (crc_route_scores), CRC_OK if none. */
int crc_device_error(void);

/* Number of kernels the library has launched in this process. */
uint64_t crc_launch_count(void);

/* Optional per-kernel timing.  Between crc_profile_begin() and
 * crc_profile_end(), every kernel the library launches is bracketed by two
 * CUDA events recorded on its launching stream.  crc_profile_end()
 * synchronises those events and returns, per kernel kind, the number of
 * launches and their summed device time in milliseconds.  Host-side
 * bookkeeping only; off by default.  Not thread-safe against concurrent
 * library calls from other host threads. */
enum { CRC_KERNEL_ROUTER = 0, CRC_KERNEL_SCAN = 1, CRC_KERNEL_STATE = 2, CRC_KERNEL_SYNTH = 3,
       CRC_KERNEL_FUSED = 4, CRC_KERNEL_LOSS = 5, CRC_KERNEL_LOSS_MEANS = 6,
       CRC_KERNEL_KINDS = 8 };
typedef struct crc_kernel_times {
    uint64_t launches[CRC_KERNEL_KINDS];
    double ms[CRC_KERNEL_KINDS];
} crc_kernel_times;
int crc_profile_begin(void);
int crc_profile_end(crc_kernel_times *out);

/* Message for an error code (static string). */
const char *crc_strerror(int code);

/* Seeded synthetic inputs (not part of the method).  Same definition as the
 * host generator: Philox4x32-10 counters, Irwin-Hall(4) unit normals,
 * separable AR(1) over layers then tokens, bf16 round-to-nearest-even.
 * crc_synth_hidden writes tokens [t0, t0 + T) of hidden bf16 [B][T][L][d]
 * (the chunk); carry_dev fp32 [B][L][d] holds h of token t0 - 1 on entry
 * (ignored when t0 == 0) and of token t0 + T - 1 on exit.  attempts_dev
 * (uint8 [B][T][L], may be NULL) selects re-drawn innovations per unit.
 * crc_synth_weights writes W_cat bf16 [L][3N][d] ~ N(0, 1/d); copy_init
 * copies native rows into the other heads (W^T_l = W^R_l,
 * W^S_l = W^R_{(l+1) mod L}). */
int crc_synth_hidden(int32_t B, int32_t T, int32_t L, int32_t d, int32_t t0,
                     uint32_t seed, double rho_t, double rho_l,
                     const uint8_t *attempts_dev, uint16_t *hidden_dev,
                     float *carry_dev, void *stream);
int crc_synth_weights(int32_t L, int32_t N, int32_t d, uint32_t seed, int32_t copy_init,
                      uint16_t *w_cat_dev, void *stream);

#ifdef __cplusplus
}
#endif
#endif /* CRC_H */
