// C-ABI entry points of the library (declared in include/crc.h): argument
// validation, state handling and the route-and-cache driver.
#include <sys/mman.h>

#include <atomic>
#include <cmath>
#include <cstdio>
#include <cstring>
#include <map>
#include <mutex>
#include <vector>

#include "crc_device.cuh"
#include "crc_internal.h"

namespace crc {
namespace {

std::atomic<uint64_t> g_launches{0};
__device__ uint32_t g_device_error;

bool aligned(const void* p, size_t a) { return (reinterpret_cast<uintptr_t>(p) % a) == 0; }

// Common problem checks; router = the limits of the router entry points.
int check_problem(const crc_problem* p, bool router) {
    if (!p) return CRC_EINVAL;
    if (p->reserved != 0) return CRC_EINVAL;
    if (p->L < 1 || p->B < 1 || p->N < 1 || p->K < 1 || p->C < 1 || p->R < 0 || p->d < 1)
        return CRC_EINVAL;
    if (p->N % 16 != 0 || p->N > 256) return CRC_EUNSUPPORTED;
    if (router && (p->N > 128 || p->d % 8 != 0)) return CRC_EUNSUPPORTED;
    if (p->K > 32 || p->K > p->C || p->C > p->N || p->R > p->N) return CRC_EUNSUPPORTED;
    const StateLayout lay = state_layout(p->B, p->L, p->N);
    if ((double)p->B * p->L > 2.0e9 || lay.total == 0) return CRC_EUNSUPPORTED;
    return CRC_OK;
}

int check_state(const crc_problem* p, const void* state, size_t bytes) {
    if (!state || !aligned(state, 256)) return CRC_EINVAL;
    if (bytes < state_layout(p->B, p->L, p->N).total) return CRC_ESTATE;
    return CRC_OK;
}

int check_trace(const crc_trace* tr) {
    // every trace pointer may be null; bytes need no alignment, mask words 4 bytes
    if (tr && ((tr->cache_mid_dev && !aligned(tr->cache_mid_dev, 4)) ||
               (tr->cache_after_dev && !aligned(tr->cache_after_dev, 4)) ||
               (tr->topk_set_dev && !aligned(tr->topk_set_dev, 4))))
        return CRC_EINVAL;
    return CRC_OK;
}

struct ProfRecord {
    int kind;
    cudaEvent_t start, stop;
};
std::mutex g_prof_mu;
bool g_prof_on = false;
std::vector<ProfRecord> g_prof;
std::vector<cudaEvent_t> g_event_pool;

cudaEvent_t pool_event() {
    if (!g_event_pool.empty()) {
        cudaEvent_t e = g_event_pool.back();
        g_event_pool.pop_back();
        return e;
    }
    cudaEvent_t e = nullptr;
    if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
    return e;
}

}  // namespace

ProfScope::ProfScope(int kind, cudaStream_t s) : slot(-1), stream(s) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    if (!g_prof_on || kind < 0 || kind >= CRC_KERNEL_KINDS) return;
    ProfRecord r{kind, pool_event(), pool_event()};
    if (!r.start || !r.stop) return;
    cudaEventRecord(r.start, s);
    slot = (int)g_prof.size();
    g_prof.push_back(r);
}

ProfScope::~ProfScope() {
    if (slot < 0) return;
    std::lock_guard<std::mutex> lk(g_prof_mu);
    cudaEventRecord(g_prof[slot].stop, stream);
}

void note_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

uint32_t* device_error_word() {
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_device_error) != cudaSuccess) return nullptr;
    return static_cast<uint32_t*>(p);
}

int sm_count() {
    int dev = 0;
    cudaGetDevice(&dev);
    static std::mutex mu;
    static std::vector<int> cache;
    std::lock_guard<std::mutex> lk(mu);
    if ((int)cache.size() <= dev) cache.resize(dev + 1, 0);
    if (cache[dev] == 0) {
        int n = 0;
        cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
        cache[dev] = n > 0 ? n : 1;
    }
    return cache[dev];
}

}  // namespace crc

using namespace crc;

extern "C" {

size_t crc_state_bytes(const crc_problem* p) {
    if (check_problem(p, false) != CRC_OK) return 0;
    return state_layout(p->B, p->L, p->N).total;
}

int crc_state_init(const crc_problem* p, void* state_dev, size_t state_bytes, void* stream) {
    int rc = check_problem(p, false);
    if (rc) return rc;
    if ((rc = check_state(p, state_dev, state_bytes))) return rc;
    return launch_state_init(*p, state_dev, state_layout(p->B, p->L, p->N).total,
                             static_cast<cudaStream_t>(stream));
}

int crc_state_read(const crc_problem* p, const void* state_dev, size_t state_bytes,
                   crc_stats* out, uint32_t* cache_bits_host, float* retention_host,
                   uint64_t* chain_counters_host, void* stream) {
    int rc = check_problem(p, false);
    if (rc) return rc;
    if ((rc = check_state(p, state_dev, state_bytes))) return rc;
    if (!out) return CRC_EINVAL;
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess)
        return CRC_ECUDA;
    const StateLayout lay = state_layout(p->B, p->L, p->N);
    const uint8_t* base = static_cast<const uint8_t*>(state_dev);
    StateHeader h;
    if (cudaMemcpy(&h, base, sizeof h, cudaMemcpyDeviceToHost) != cudaSuccess) return CRC_ECUDA;
    if (h.magic != kStateMagic || h.L != p->L || h.N != p->N || h.K != p->K || h.C != p->C ||
        h.R != p->R || h.B != p->B)
        return CRC_ESTATE;
    const size_t nchains = (size_t)p->B * p->L;
    std::vector<ChainState> ch(nchains);
    if (cudaMemcpy(ch.data(), base + lay.chains, nchains * sizeof(ChainState),
                   cudaMemcpyDeviceToHost) != cudaSuccess)
        return CRC_ECUDA;
    std::memset(out, 0, sizeof *out);
    const int NW = (p->N + 31) / 32;
    for (size_t c = 0; c < nchains; ++c) {
        out->hits += ch[c].hits;
        out->misses += ch[c].misses;
        out->proactive += ch[c].proactive;
        if (cache_bits_host)
            for (int w = 0; w < NW; ++w) cache_bits_host[c * NW + w] = ch[c].bits[w];
        if (chain_counters_host) {
            chain_counters_host[c * 3 + 0] = ch[c].hits;
            chain_counters_host[c * 3 + 1] = ch[c].misses;
            chain_counters_host[c * 3 + 2] = ch[c].proactive;
        }
    }
    out->accesses = out->hits + out->misses;
    out->traffic_bytes = (out->misses + out->proactive) * p->expert_bytes;
    out->tokens = (uint64_t)h.t_next;
    out->error = h.error;
    if (retention_host &&
        cudaMemcpy(retention_host, base + lay.retention, nchains * p->N * sizeof(float),
                   cudaMemcpyDeviceToHost) != cudaSuccess)
        return CRC_ECUDA;
    return h.error ? (int)h.error : CRC_OK;
}

int crc_metrics(const crc_problem* p, const crc_stats* s, crc_report* out) {
    if (!s || !out || check_problem(p, false) != CRC_OK) return CRC_EINVAL;
    const double A = (double)s->accesses, D = (double)s->misses, P = (double)s->proactive;
    const double tokens = (double)p->B * (double)s->tokens;
    const double moved = (D + P) * (double)p->expert_bytes;
    out->hit = A > 0.0 ? 1.0 - D / A : NAN;
    out->adj_hit = A + P > 0.0 ? (A - D) / (A + P) : NAN;
    out->traffic_bytes = moved;
    out->load_per_token_bytes = tokens > 0.0 ? moved / tokens : 0.0;
    return CRC_OK;
}

int crc_load_time(const crc_problem* p, const crc_stats* s, double c_exp, double eta,
                  double* t_load) {
    if (!s || !t_load || check_problem(p, false) != CRC_OK) return CRC_EINVAL;
    if (!(eta >= 0.0 && eta <= 1.0) || !(c_exp >= 0.0) || !std::isfinite(c_exp))
        return CRC_EINVAL;
    const double tokens = (double)p->B * (double)s->tokens;
    *t_load = tokens > 0.0
                  ? c_exp / tokens * ((double)s->misses + (1.0 - eta) * (double)s->proactive)
                  : 0.0;
    return CRC_OK;
}

int crc_route_scores(const crc_problem* p, const uint16_t* hidden_dev, const uint16_t* w_cat_dev,
                     int32_t T, int32_t heads, float* scores_dev, void* stream) {
    int rc = check_problem(p, true);
    if (rc) return rc;
    if (T < 0 || (heads != 2 && heads != 3)) return CRC_EINVAL;
    if (T == 0) return CRC_OK;
    if (!hidden_dev || !w_cat_dev || !scores_dev) return CRC_EINVAL;
    if (!aligned(hidden_dev, 16) || !aligned(w_cat_dev, 16) || !aligned(scores_dev, 16))
        return CRC_EINVAL;
    return launch_router(*p, hidden_dev, T, 0, T, w_cat_dev, heads, scores_dev,
                         device_error_word(), static_cast<cudaStream_t>(stream));
}

int crc_cache_scan(const crc_problem* p, const float* scores_dev, int32_t T, void* state_dev,
                   size_t state_bytes, const crc_trace* trace, void* stream) {
    int rc = check_problem(p, false);
    if (rc) return rc;
    if ((rc = check_state(p, state_dev, state_bytes))) return rc;
    if (T < 0) return CRC_EINVAL;
    if (T == 0) return CRC_OK;
    if (!scores_dev || !aligned(scores_dev, 16)) return CRC_EINVAL;
    if ((rc = check_trace(trace))) return rc;
    return launch_scan(*p, scores_dev, T, state_dev, trace, T, 0,
                       static_cast<cudaStream_t>(stream));
}

int crc_cache_scan_policy(const crc_problem* p, const float* scores_dev, int32_t T,
                          void* state_dev, size_t state_bytes, const crc_trace* trace,
                          int32_t policy, int32_t lambda_halves, void* stream) {
    int rc = check_problem(p, false);
    if (rc) return rc;
    if ((rc = check_state(p, state_dev, state_bytes))) return rc;
    if (policy < CRC_POLICY_LRU || policy > CRC_POLICY_SPATIO_LRU) return CRC_EINVAL;
    if (lambda_halves < 0 || lambda_halves > 8) return CRC_EINVAL;
    if (T < 0) return CRC_EINVAL;
    if (T == 0) return CRC_OK;
    if (!scores_dev || !aligned(scores_dev, 16)) return CRC_EINVAL;
    if ((rc = check_trace(trace))) return rc;
    return launch_policy_scan(*p, scores_dev, T, state_dev, trace, T, 0, policy, lambda_halves,
                              static_cast<cudaStream_t>(stream));
}

int crc_state_read_aux(const crc_problem* p, const void* state_dev, size_t state_bytes,
                       uint32_t* aux_host, void* stream) {
    int rc = check_problem(p, false);
    if (rc) return rc;
    if ((rc = check_state(p, state_dev, state_bytes))) return rc;
    if (!aux_host) return CRC_EINVAL;
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return CRC_ECUDA;
    const StateLayout lay = state_layout(p->B, p->L, p->N);
    const uint8_t* base = static_cast<const uint8_t*>(state_dev);
    if (cudaMemcpy(aux_host, base + lay.aux, (size_t)p->B * p->L * p->N * sizeof(uint32_t),
                   cudaMemcpyDeviceToHost) != cudaSuccess)
        return CRC_ECUDA;
    return CRC_OK;
}

size_t crc_fused_workspace_bytes(const crc_problem* p) {
    if (check_problem(p, true) != CRC_OK) return 0;
    return fused_workspace_bytes(*p);
}

size_t crc_workspace_bytes(const crc_problem* p, int32_t chunk_tokens) {
    if (check_problem(p, true) != CRC_OK || chunk_tokens < 1) return 0;
    return (size_t)p->B * chunk_tokens * p->L * 3 * p->N * sizeof(float);
}

int crc_route_and_cache(const crc_problem* p, const uint16_t* hidden_dev,
                        const uint16_t* w_cat_dev, int32_t T, void* state_dev,
                        size_t state_bytes, const crc_trace* trace, void* workspace_dev,
                        size_t workspace_bytes, void* stream) {
    int rc = check_problem(p, true);
    if (rc) return rc;
    if ((rc = check_state(p, state_dev, state_bytes))) return rc;
    if (T < 0) return CRC_EINVAL;
    if (T == 0) return CRC_OK;
    if (!hidden_dev || !w_cat_dev || !aligned(hidden_dev, 16) || !aligned(w_cat_dev, 16))
        return CRC_EINVAL;
    if (!workspace_dev || !aligned(workspace_dev, 256)) return CRC_EINVAL;
    if ((rc = check_trace(trace))) return rc;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    // the fused kernel knows the Top-K as a set only: a trace in rank order
    // takes the two-kernel path
    if (!(trace && trace->topk_dev)) {
        rc = launch_fused(*p, hidden_dev, w_cat_dev, T, state_dev, workspace_dev, workspace_bytes,
                          trace, s);
        if (rc != CRC_EUNSUPPORTED) return rc;
    }
    const size_t per_token = crc_workspace_bytes(p, 1);
    const long long fit = (long long)(workspace_bytes / per_token);
    if (fit < 1) return CRC_EINVAL;
    const int chunk = fit < T ? (int)fit : T;
    float* scores = static_cast<float*>(workspace_dev);
    const int heads = p->R > 0 ? 3 : 2;
    uint32_t* err = static_cast<uint32_t*>(state_dev) + 1;   // StateHeader::error
    for (int t0 = 0; t0 < T; t0 += chunk) {
        const int n = (T - t0) < chunk ? (T - t0) : chunk;
        if ((rc = launch_router(*p, hidden_dev, T, t0, n, w_cat_dev, heads, scores, err, s)))
            return rc;
        if ((rc = launch_scan(*p, scores, n, state_dev, trace, T, t0, s))) return rc;
    }
    return CRC_OK;
}

size_t crc_host_staging_bytes(const crc_problem* p, int32_t chunk_tokens) {
    if (check_problem(p, true) != CRC_OK || chunk_tokens < 1) return 0;
    const size_t half = (size_t)p->B * chunk_tokens * p->L * p->d * sizeof(uint16_t);
    return 2 * ((half + 255) / 256 * 256);
}

int crc_route_and_cache_host(const crc_problem* p, const uint16_t* hidden_host,
                             const uint16_t* w_cat_dev, int32_t T, int32_t chunk_tokens,
                             void* state_dev, size_t state_bytes, void* staging_dev,
                             size_t staging_bytes, void* workspace_dev, size_t workspace_bytes,
                             void* stream) {
    int rc = check_problem(p, true);
    if (rc) return rc;
    if ((rc = check_state(p, state_dev, state_bytes))) return rc;
    if (T < 0 || chunk_tokens < 1) return CRC_EINVAL;
    if (T == 0) return CRC_OK;
    if (!hidden_host || !aligned(hidden_host, 16) || !w_cat_dev || !aligned(w_cat_dev, 16))
        return CRC_EINVAL;
    const int chunk = chunk_tokens < T ? chunk_tokens : T;
    if (!staging_dev || !aligned(staging_dev, 256) ||
        staging_bytes < crc_host_staging_bytes(p, chunk))
        return CRC_EINVAL;
    if (!workspace_dev || !aligned(workspace_dev, 256)) return CRC_EINVAL;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const size_t row = (size_t)p->L * p->d * sizeof(uint16_t);        // one token of one stream
    const size_t half = crc_host_staging_bytes(p, chunk) / 2;
    int max_pitch = 0, dev = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&max_pitch, cudaDevAttrMaxPitch, dev);
    const bool two_d = (double)T * row <= (double)max_pitch;

    // Copies run on a stream of the call's own, chunk i into staging half i % 2,
    // while `stream` runs the step on chunk i - 1.  copied[j]: half j holds its
    // chunk; done[j]: the step that read half j has finished with it.
    cudaStream_t cs = nullptr;
    cudaEvent_t entry = nullptr, joined = nullptr, copied[2] = {nullptr, nullptr},
                done[2] = {nullptr, nullptr};
    bool ok = cudaStreamCreateWithFlags(&cs, cudaStreamNonBlocking) == cudaSuccess;
    for (cudaEvent_t* e : {&entry, &joined, &copied[0], &copied[1], &done[0], &done[1]})
        ok = ok && cudaEventCreateWithFlags(e, cudaEventDisableTiming) == cudaSuccess;
    // the staging halves may still be read by work queued earlier on `stream`
    ok = ok && cudaEventRecord(entry, s) == cudaSuccess &&
         cudaStreamWaitEvent(cs, entry, 0) == cudaSuccess;
    rc = ok ? CRC_OK : CRC_ECUDA;
    for (int t0 = 0, i = 0; rc == CRC_OK && t0 < T; t0 += chunk, ++i) {
        const int n = (T - t0) < chunk ? (T - t0) : chunk;
        const int j = i & 1;
        uint8_t* buf = static_cast<uint8_t*>(staging_dev) + (size_t)j * half;
        const uint8_t* src = reinterpret_cast<const uint8_t*>(hidden_host) + (size_t)t0 * row;
        if (i >= 2 && cudaStreamWaitEvent(cs, done[j], 0) != cudaSuccess) rc = CRC_ECUDA;
        // [B][n][L][d] of the chunk, stream b's tokens at pitch T * row in host memory
        if (rc == CRC_OK && two_d) {
            if (cudaMemcpy2DAsync(buf, (size_t)n * row, src, (size_t)T * row, (size_t)n * row,
                                  (size_t)p->B, cudaMemcpyHostToDevice, cs) != cudaSuccess)
                rc = CRC_ECUDA;
        } else {
            for (int b = 0; rc == CRC_OK && b < p->B; ++b)
                if (cudaMemcpyAsync(buf + (size_t)b * n * row, src + (size_t)b * T * row,
                                    (size_t)n * row, cudaMemcpyHostToDevice, cs) != cudaSuccess)
                    rc = CRC_ECUDA;
        }
        if (rc == CRC_OK && (cudaEventRecord(copied[j], cs) != cudaSuccess ||
                             cudaStreamWaitEvent(s, copied[j], 0) != cudaSuccess))
            rc = CRC_ECUDA;
        if (rc == CRC_OK)
            rc = crc_route_and_cache(p, reinterpret_cast<const uint16_t*>(buf), w_cat_dev, n,
                                     state_dev, state_bytes, nullptr, workspace_dev,
                                     workspace_bytes, stream);
        if (rc == CRC_OK && cudaEventRecord(done[j], s) != cudaSuccess) rc = CRC_ECUDA;
    }
    // everything the call queued on its copy stream is ordered before later work on `stream`
    if (cs && joined && cudaEventRecord(joined, cs) == cudaSuccess)
        cudaStreamWaitEvent(s, joined, 0);
    for (cudaEvent_t e : {entry, joined, copied[0], copied[1], done[0], done[1]})
        if (e) cudaEventDestroy(e);
    if (cs) cudaStreamDestroy(cs);
    return rc;
}

// Pinned host memory on transparent huge pages: anonymous mappings aligned to
// the kernel's huge-page size, advised MADV_HUGEPAGE, faulted in one huge page
// at a time and registered with CUDA.  The registry maps the pointer handed
// out to its mapping.
namespace {
struct HostMapping {
    void* base;
    size_t len;
};
std::mutex g_host_mu;
std::map<uintptr_t, HostMapping> g_host_maps;

size_t huge_page_bytes() {
    size_t hp = 2u << 20;
    if (FILE* f = std::fopen("/sys/kernel/mm/transparent_hugepage/hpage_pmd_size", "r")) {
        unsigned long long v = 0;
        if (std::fscanf(f, "%llu", &v) == 1 && v >= 4096 && (v & (v - 1)) == 0) hp = (size_t)v;
        std::fclose(f);
    }
    return hp;
}
}  // namespace

int crc_host_alloc(size_t bytes, void** out) {
    if (!out) return CRC_EINVAL;
    *out = nullptr;
    if (bytes == 0) return CRC_EINVAL;
    const size_t hp = huge_page_bytes();
    const size_t body = (bytes + hp - 1) / hp * hp;
    if (body < bytes || body + hp < body) return CRC_EINVAL;
    const size_t len = body + hp;
    void* base = mmap(nullptr, len, PROT_READ | PROT_WRITE, MAP_PRIVATE | MAP_ANONYMOUS, -1, 0);
    if (base == MAP_FAILED) return CRC_ENOMEM;
    uint8_t* p = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(base) + hp - 1) / hp * hp);
#ifdef MADV_HUGEPAGE
    madvise(p, body, MADV_HUGEPAGE);    // advisory: base pages if huge pages are unavailable
#endif
    for (size_t o = 0; o < body; o += hp) p[o] = 0;
    if (cudaHostRegister(p, body, cudaHostRegisterDefault) != cudaSuccess) {
        cudaGetLastError();
        munmap(base, len);
        return CRC_ECUDA;
    }
    {
        std::lock_guard<std::mutex> lk(g_host_mu);
        g_host_maps[reinterpret_cast<uintptr_t>(p)] = HostMapping{base, len};
    }
    *out = p;
    return CRC_OK;
}

int crc_host_free(void* ptr) {
    if (!ptr) return CRC_OK;
    HostMapping m;
    {
        std::lock_guard<std::mutex> lk(g_host_mu);
        auto it = g_host_maps.find(reinterpret_cast<uintptr_t>(ptr));
        if (it == g_host_maps.end()) return CRC_EINVAL;
        m = it->second;
        g_host_maps.erase(it);
    }
    const int rc = cudaHostUnregister(ptr) == cudaSuccess ? CRC_OK : CRC_ECUDA;
    munmap(m.base, m.len);
    return rc;
}

size_t crc_loss_workspace_bytes(const crc_problem* p, int32_t T) {
    if (check_problem(p, false) != CRC_OK || T < 1) return 0;
    const size_t bytes = (size_t)loss_task_slots(p->B, p->L, T, p->N) * 2 * sizeof(double);
    return (bytes + 255) / 256 * 256;
}

int crc_cache_loss(const crc_problem* p, const float* probs_dev, int32_t T, int32_t heads,
                   int32_t top_b, double tau, double w_T, double w_ST, float* loss_dev,
                   double* means_dev, float* grad_dev, void* workspace_dev,
                   size_t workspace_bytes, void* stream) {
    int rc = check_problem(p, false);
    if (rc) return rc;
    if (T < 0 || (heads != 2 && heads != 3)) return CRC_EINVAL;
    if (top_b < 1 || top_b > p->N) return CRC_EINVAL;
    if (!(tau > 0.0) || !std::isfinite(tau) || !std::isfinite(1.0 / tau)) return CRC_EINVAL;
    if (!std::isfinite(w_T) || !std::isfinite(w_ST)) return CRC_EINVAL;
    if (T == 0) return CRC_OK;
    if (!probs_dev || !aligned(probs_dev, 16)) return CRC_EINVAL;
    if (grad_dev && (!aligned(grad_dev, 16) || (const void*)grad_dev == (const void*)probs_dev))
        return CRC_EINVAL;
    if (loss_dev && !aligned(loss_dev, 4)) return CRC_EINVAL;
    if (means_dev) {
        if (!aligned(means_dev, 8) || !workspace_dev || !aligned(workspace_dev, 256) ||
            workspace_bytes < crc_loss_workspace_bytes(p, T))
            return CRC_EINVAL;
    }
    if (!loss_dev && !means_dev && !grad_dev) return CRC_OK;
    return launch_cache_loss(*p, probs_dev, T, heads, top_b, tau, w_T, w_ST, loss_dev, means_dev,
                             grad_dev, workspace_dev, static_cast<cudaStream_t>(stream));
}

int crc_device_error(void) {
    if (cudaDeviceSynchronize() != cudaSuccess) return CRC_ECUDA;
    uint32_t v = 0, zero = 0;
    if (cudaMemcpyFromSymbol(&v, g_device_error, sizeof v) != cudaSuccess) return CRC_ECUDA;
    if (cudaMemcpyToSymbol(g_device_error, &zero, sizeof zero) != cudaSuccess) return CRC_ECUDA;
    return (int)v;
}

uint64_t crc_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

int crc_profile_begin(void) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    for (auto& r : g_prof) {
        g_event_pool.push_back(r.start);
        g_event_pool.push_back(r.stop);
    }
    g_prof.clear();
    g_prof_on = true;
    return CRC_OK;
}

int crc_profile_end(crc_kernel_times* out) {
    std::lock_guard<std::mutex> lk(g_prof_mu);
    g_prof_on = false;
    if (out) std::memset(out, 0, sizeof *out);
    int rc = CRC_OK;
    for (auto& r : g_prof) {
        float ms = 0.f;
        if (cudaEventSynchronize(r.stop) != cudaSuccess ||
            cudaEventElapsedTime(&ms, r.start, r.stop) != cudaSuccess) {
            rc = CRC_ECUDA;
            continue;
        }
        if (out) {
            out->launches[r.kind] += 1;
            out->ms[r.kind] += ms;
        }
    }
    return rc;
}

const char* crc_strerror(int code) {
    switch (code) {
        case CRC_OK: return "ok";
        case CRC_EINVAL: return "invalid argument (null or misaligned pointer, bad size)";
        case CRC_EUNSUPPORTED: return "sizes outside the supported limits";
        case CRC_ECUDA: return "CUDA runtime error";
        case CRC_ETIMEOUT: return "a bounded device wait ran out";
        case CRC_ESTATE: return "state buffer too small, uninitialised or for another problem";
        case CRC_EDEVICE: return "device-side failure";
        case CRC_ENOMEM: return "out of host memory";
        default: return "unknown error code";
    }
}

int crc_synth_hidden(int32_t B, int32_t T, int32_t L, int32_t d, int32_t t0, uint32_t seed,
                     double rho_t, double rho_l, const uint8_t* attempts_dev,
                     uint16_t* hidden_dev, float* carry_dev, void* stream) {
    if (B < 1 || T < 0 || L < 1 || d < 2 || d % 2 || t0 < 0) return CRC_EINVAL;
    if (!(rho_t >= 0.0 && rho_t <= 1.0 && rho_l >= 0.0 && rho_l <= 1.0)) return CRC_EINVAL;
    if (T == 0) return CRC_OK;
    if (!hidden_dev || !carry_dev || !aligned(hidden_dev, 4) || !aligned(carry_dev, 8))
        return CRC_EINVAL;
    return launch_synth_hidden(B, T, L, d, t0, seed, rho_t, rho_l, attempts_dev, hidden_dev,
                               carry_dev, static_cast<cudaStream_t>(stream));
}

int crc_synth_weights(int32_t L, int32_t N, int32_t d, uint32_t seed, int32_t copy_init,
                      uint16_t* w_cat_dev, void* stream) {
    if (L < 1 || N < 1 || d < 2 || d % 2) return CRC_EINVAL;
    if (!w_cat_dev || !aligned(w_cat_dev, 4)) return CRC_EINVAL;
    return launch_synth_weights(L, N, d, seed, copy_init ? 1 : 0, w_cat_dev,
                                static_cast<cudaStream_t>(stream));
}

}  // extern "C"
