// Expert transfer engine: the cache simulation's load decisions as copies of
// expert weights from a host pool into a device-resident cache of C slots per
// layer (the expert pool of the problem statement, Sec. 2, and the transfers
// counted by the Sec. 4.1 metrics).
//
// Planning (host only): one stream's trace gives, per access, the cache after
// Algorithm 2's refinement and after Algorithm 1's update.  Against the cache
// before the access, the proactive loads are C~ \ C and the demand loads
// C+ \ C~; the experts that leave in a phase free their slots.  Within a phase
// the freed slots are taken first, in ascending slot order, by the loaded
// experts in ascending expert order, then the free slots.  An expert never
// enters and leaves within one phase (a refinement candidate that was
// inserted outranks every later candidate, and UpdateCache protects the
// selected experts it loads), so the plan holds exactly P + D copies.
//
// Replay: one cudaMemcpyAsync per planned copy, host pool to slot, in plan
// order on the caller's stream.
#include <cstring>
#include <vector>

#include "crc_internal.h"

namespace crc {
namespace {

inline bool bit(const uint32_t* w, int e) { return (w[e >> 5] >> (e & 31)) & 1u; }

}  // namespace
}  // namespace crc

using namespace crc;

extern "C" {

int crc_transfer_plan(const crc_problem* p, int32_t T, const uint32_t* mid_host,
                      const uint32_t* after_host, const uint32_t* start_host,
                      int32_t* slot_expert, crc_transfer* out, int64_t max_out,
                      int64_t* n_out) {
    if (!p || p->L < 1 || p->N < 1 || p->N > 256 || p->C < 1 || p->C > p->N) return CRC_EINVAL;
    if (T < 0 || !slot_expert || !n_out || max_out < 0 || (max_out > 0 && !out))
        return CRC_EINVAL;
    if (T > 0 && (!mid_host || !after_host)) return CRC_EINVAL;
    const int L = p->L, N = p->N, C = p->C, NW = (N + 31) / 32;
    // the cache before token 0 and its slot map must agree
    std::vector<uint32_t> cur((size_t)L * NW, 0u);
    for (int l = 0; l < L; ++l) {
        uint32_t* c = &cur[(size_t)l * NW];
        for (int s = 0; s < C; ++s) {
            const int e = slot_expert[(size_t)l * C + s];
            if (e < -1 || e >= N) return CRC_EINVAL;
            if (e >= 0) {
                if (bit(c, e)) return CRC_EINVAL;               // an expert in two slots
                c[e >> 5] |= 1u << (e & 31);
            }
        }
        if (start_host)
            for (int w = 0; w < NW; ++w)
                if (start_host[(size_t)l * NW + w] != c[w]) return CRC_EINVAL;
    }
    int64_t n = 0;
    std::vector<int> freed, left, loads;
    freed.reserve(C);
    left.reserve(C);
    loads.reserve(N);
    for (int t = 0; t < T; ++t) {
        for (int l = 0; l < L; ++l) {
            uint32_t* c = &cur[(size_t)l * NW];
            int32_t* map = slot_expert + (size_t)l * C;
            const size_t u = ((size_t)t * L + l) * NW;
            for (int phase = 0; phase < 2; ++phase) {
                const uint32_t* nxt = (phase == 0 ? mid_host : after_host) + u;
                freed.clear();
                left.clear();
                loads.clear();
                for (int s = 0; s < C; ++s) {
                    const int e = map[s];
                    if (e >= 0 && !bit(nxt, e)) {               // leaves the cache
                        freed.push_back(s);
                        left.push_back(e);
                        map[s] = -1;
                    }
                }
                int occupied = 0;
                for (int e = 0; e < N; ++e) {
                    if (bit(nxt, e)) {
                        ++occupied;
                        if (!bit(c, e)) loads.push_back(e);     // enters the cache
                    }
                }
                if (occupied > C) return CRC_EINVAL;            // not a C-slot cache
                size_t fi = 0;
                int free_cursor = 0;
                for (int e : loads) {
                    int s, gone = -1;
                    if (fi < freed.size()) {
                        gone = left[fi];
                        s = freed[fi++];
                    } else {
                        while (free_cursor < C && map[free_cursor] >= 0) ++free_cursor;
                        s = free_cursor;                        // occupied <= C: one exists
                    }
                    if (n < max_out) {
                        crc_transfer& x = out[n];
                        x.t = t;
                        x.l = l;
                        x.expert = e;
                        x.slot = s;
                        x.evicted = gone;
                        x.proactive = phase == 0 ? 1 : 0;
                    }
                    map[s] = e;
                    ++n;
                }
                for (int w = 0; w < NW; ++w) c[w] = nxt[w];
            }
        }
    }
    *n_out = n;
    return (out && n > max_out) ? CRC_EINVAL : CRC_OK;   // out = NULL: count only
}

int crc_transfer_replay(const crc_problem* p, const crc_transfer* plan, int64_t n,
                        const void* pool_host, int64_t pool_experts, void* slots_dev,
                        void* stream) {
    if (!p || p->L < 1 || p->N < 1 || p->C < 1 || p->expert_bytes == 0) return CRC_EINVAL;
    if (n < 0 || (n > 0 && (!plan || !pool_host || !slots_dev)) || pool_experts < 1)
        return CRC_EINVAL;
    const size_t eb = (size_t)p->expert_bytes;
    const int L = p->L, N = p->N, C = p->C;
    for (int64_t i = 0; i < n; ++i) {
        const crc_transfer& x = plan[i];
        if (x.l < 0 || x.l >= L || x.expert < 0 || x.expert >= N || x.slot < 0 || x.slot >= C)
            return CRC_EINVAL;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const uint8_t* pool = static_cast<const uint8_t*>(pool_host);
    uint8_t* slots = static_cast<uint8_t*>(slots_dev);
    for (int64_t i = 0; i < n; ++i) {
        const crc_transfer& x = plan[i];
        const int64_t src = ((int64_t)x.l * N + x.expert) % pool_experts;
        if (cudaMemcpyAsync(slots + ((size_t)x.l * C + x.slot) * eb, pool + (size_t)src * eb, eb,
                            cudaMemcpyHostToDevice, s) != cudaSuccess)
            return CRC_ECUDA;
    }
    return CRC_OK;
}

}  // extern "C"
