// Cache scan: one warp per (stream, layer) chain, sequential over tokens.
//
// Lane i owns experts [i*V, i*V + V).  Per access (Algorithm 2 of the paper
// with Algorithm 1 as its last step):
//   s^T  = p^R + p^T                                   (Sec. 3.2)
//   s^ST = s^T_{t-1} + p^S_{rho(t,l)}  (R > 0, t >= 1)  (Sec. 3.3)
//   refinement over A = Top_R(s^ST): skip residents, fill a free slot,
//   else replace the lowest resident when strictly higher; a candidate that
//   loses ends the refinement (every later one is no higher and the lowest
//   resident only rises, so it would lose too);
//   S = TopK(p^R); misses = |S \ C~|;
//   UpdateCache: demand-loaded experts fill free slots, then each further one
//   evicts the lowest-s^T resident outside S (the demand set's order does not
//   change the resulting set, since inserted experts are in S and protected).
// Reductions: the fp32 bit patterns of the (non-negative) scores serve as
// ordered 32-bit keys.  Each lane keeps its keys sorted in policy order, so a
// warp-wide "first in order" is one redux.sync (max key) and a ballot whose
// lowest set lane owns it; a "last member" is a lane-local scan, a
// redux.sync (min key) and a ballot whose highest set lane owns it.  Only the
// owner lane learns which of its experts was picked.
#pragma once

#include "crc_device.cuh"

namespace crc {

struct ScanArgs {
    const float* scores;     // [B][T][L][3][N]
    uint8_t* state;          // state buffer base
    uint8_t* trace_topk;     // [B][T][L][K] or null
    uint8_t* trace_miss;     // [B][T][L] or null
    uint8_t* trace_pro;      // [B][T][L] or null
    uint32_t* trace_mid;     // [B][T][L][NW] cache after the refinement, or null
    uint32_t* trace_after;   // [B][T][L][NW] cache after UpdateCache, or null
    uint32_t* trace_sel;     // [B][T][L][NW] native Top-K set, or null
    int trace_T, trace_t0;   // trace arrays span trace_T tokens; this call starts at trace_t0
    int B, T, L, N, K, C, R;
};

// Keys: scores are non-negative, so their fp32 bit patterns are already
// ordered like the values; +1 keeps every real key above 0, which marks an
// empty slot.  Each lane keeps (key, slot) pairs sorted in policy order
// (key descending, equal keys by ascending slot = ascending expert index).
__device__ __forceinline__ uint32_t pkey(float x) { return __float_as_uint(x) + 1u; }
__device__ __forceinline__ uint32_t umin(uint32_t a, uint32_t b) { return a < b ? a : b; }
__device__ __forceinline__ uint32_t umax(uint32_t a, uint32_t b) { return a > b ? a : b; }

template <int V>
struct KeyList {
    uint32_t k[V];
    uint32_t s[V];
};

// Stable sort of a lane's V entries: odd-even transposition that swaps only
// strictly smaller keys forward, so equal keys keep their ascending slots.
template <int V>
__device__ __forceinline__ void presort(KeyList<V>& L) {
#pragma unroll
    for (int round = 0; round < V; ++round) {
#pragma unroll
        for (int j = round & 1; j + 1 < V; j += 2) {
            const bool sw = L.k[j + 1] > L.k[j];
            const uint32_t k0 = L.k[j], s0 = L.s[j];
            L.k[j] = sw ? L.k[j + 1] : k0;
            L.s[j] = sw ? L.s[j + 1] : s0;
            L.k[j + 1] = sw ? k0 : L.k[j + 1];
            L.s[j + 1] = sw ? s0 : L.s[j + 1];
        }
    }
}

// Removes the warp-wide first entry in policy order: the largest head key and,
// among lanes whose head has it, the lowest lane (lanes own ascending index
// ranges; a lane's head is its lowest index among equal keys).  Returns the
// owner lane (-1 when every list is empty); the owner receives the slot.
template <int V>
__device__ __forceinline__ int warp_pop_first(KeyList<V>& L, int lane, uint32_t& key,
                                              uint32_t& slot) {
    const uint32_t m = __reduce_max_sync(kFull, L.k[0]);
    key = m;
    const uint32_t b = __ballot_sync(kFull, m != 0u && L.k[0] == m);
    if (b == 0u) return -1;
    const int owner = __ffs(b) - 1;
    if (lane == owner) {
        slot = L.s[0];
#pragma unroll
        for (int j = 0; j + 1 < V; ++j) {
            L.k[j] = L.k[j + 1];
            L.s[j] = L.s[j + 1];
        }
        L.k[V - 1] = 0u;
    }
    return owner;
}

// Last member in policy order among the slots flagged in `members`: smallest
// key and, among equal keys, the highest index.  Returns the owner lane (-1 if
// no member); the owner receives the slot.  Keys are >= 1, so a non-member
// counts as the largest key, 0xffffffff, which no real key reaches.
template <int V>
__device__ __forceinline__ int warp_last_member(const uint32_t (&k)[V], uint32_t members,
                                                int lane, uint32_t& key, uint32_t& slot) {
    uint32_t m[V];
#pragma unroll
    for (int v = 0; v < V; ++v) m[v] = ((members >> v) & 1u) ? k[v] : 0xffffffffu;
    uint32_t best = m[0];
#pragma unroll
    for (int v = 1; v < V; ++v) best = umin(best, m[v]);
    const uint32_t mn = __reduce_min_sync(kFull, best);
    key = mn;
    const uint32_t b = __ballot_sync(kFull, best == mn);
    if (mn == 0xffffffffu) return -1;
    const int owner = 31 - __clz(b);
    uint32_t bs = 0u;
#pragma unroll
    for (int v = 0; v < V; ++v) bs = m[v] == mn ? (uint32_t)v : bs;   // the highest such slot
    if (lane == owner) slot = bs;
    return owner;
}

template <int V>
struct Vec {
    float v[V];
};

template <int V>
__device__ __forceinline__ Vec<V> load_vec(const float* p, bool ok) {
    Vec<V> r;
    if (!ok) {
#pragma unroll
        for (int i = 0; i < V; ++i) r.v[i] = 0.f;
        return r;
    }
    if constexpr (V == 4) {
        const float4 x = __ldg(reinterpret_cast<const float4*>(p));
        r.v[0] = x.x; r.v[1] = x.y; r.v[2] = x.z; r.v[3] = x.w;
    } else if constexpr (V == 2) {
        const float2 x = __ldg(reinterpret_cast<const float2*>(p));
        r.v[0] = x.x; r.v[1] = x.y;
    } else if constexpr (V == 8) {
        const float4 x = __ldg(reinterpret_cast<const float4*>(p));
        const float4 y = __ldg(reinterpret_cast<const float4*>(p) + 1);
        r.v[0] = x.x; r.v[1] = x.y; r.v[2] = x.z; r.v[3] = x.w;
        r.v[4] = y.x; r.v[5] = y.y; r.v[6] = y.z; r.v[7] = y.w;
    } else {
        r.v[0] = __ldg(p);
    }
    return r;
}

// Chain-local state held in registers across tokens.
template <int V>
struct ChainRegs {
    uint32_t cache;      // V bits: residency of this lane's experts
    int count;           // |C| (warp-uniform)
    float aT[V];         // s^T of the previous token
    uint32_t hits, misses, pro;
};

// ---------------------------------------------------------------------------
// Thread-serial Top-K set of one score row (used for many tokens at once, one
// token per lane).  Sorting networks on fp32 values (max/min only) find the
// K-th largest value theta; a second pass in index order takes every value
// above theta and, among values equal to theta, the lowest indices -- exactly
// the first K under (score desc, index asc).
// ---------------------------------------------------------------------------
constexpr int pow2_at_least(int x) {
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}

// Sort P values descending (P a power of two), fully unrolled: the bitonic
// network.
template <int P>
__device__ __forceinline__ void bitonic_sort_desc(float (&a)[P]) {
#pragma unroll
    for (int k = 2; k <= P; k <<= 1) {
#pragma unroll
        for (int j = k >> 1; j > 0; j >>= 1) {
#pragma unroll
            for (int i = 0; i < P; ++i) {
                const int l = i ^ j;
                if (l > i) {
                    const float hi = fmaxf(a[i], a[l]), lo = fminf(a[i], a[l]);
                    if ((i & k) == 0) {
                        a[i] = hi;
                        a[l] = lo;
                    } else {
                        a[i] = lo;
                        a[l] = hi;
                    }
                }
            }
        }
    }
}

// The same with Batcher's odd-even merge sort, which sorts P = 4 with 5
// compare-exchanges and P = 8 with 19 (the bitonic network takes 6 and 24).
// Stage p merges sorted runs of p into runs of 2p; within it, the
// compare-exchanges at distance k join elements of the same run of 2p.  Used
// up to P = 8; beyond that the compiler no longer resolves every index.
template <int P>
__device__ __forceinline__ void sort_desc(float (&a)[P]) {
    if constexpr (P > 8) {
        bitonic_sort_desc<P>(a);
    } else {
#pragma unroll
        for (int p = 1; p < P; p <<= 1) {
#pragma unroll
            for (int k = p; k >= 1; k >>= 1) {
#pragma unroll
                for (int j = k % p; j + k < P; j += 2 * k) {
#pragma unroll
                    for (int i = 0; i < k; ++i) {
                        const int x = i + j, y = i + j + k;
                        if (y < P && x / (2 * p) == y / (2 * p)) {
                            const float hi = fmaxf(a[x], a[y]), lo = fminf(a[x], a[y]);
                            a[x] = hi;
                            a[y] = lo;
                        }
                    }
                }
            }
        }
    }
}

// run <- the P largest of (run, b), both sorted descending; result descending.
template <int P>
__device__ __forceinline__ void merge_top_desc(float (&run)[P], const float (&b)[P]) {
#pragma unroll
    for (int i = 0; i < P; ++i) run[i] = fmaxf(run[i], b[P - 1 - i]);   // bitonic
#pragma unroll
    for (int j = P >> 1; j > 0; j >>= 1) {
#pragma unroll
        for (int i = 0; i < P; ++i) {
            const int l = i ^ j;
            if (l > i) {
                const float hi = fmaxf(run[i], run[l]), lo = fminf(run[i], run[l]);
                run[i] = hi;
                run[l] = lo;
            }
        }
    }
}

// Running top-KP values (descending) of a stream of non-negative scores fed 16
// at a time; theta(K) is then the K-th largest score and need(K) how many of
// the scores equal to theta belong to the Top-K set (the lowest indices).
template <int KP>
struct TopKAcc {
    float run[KP];
    __device__ __forceinline__ void init() {
#pragma unroll
        for (int i = 0; i < KP; ++i) run[i] = -1.0f;   // below every score
    }
    __device__ __forceinline__ void add16(const float* x) {
        constexpr int G = KP < 16 ? KP : 16;
#pragma unroll
        for (int g = 0; g < 16; g += G) {
            float b[KP];
#pragma unroll
            for (int i = 0; i < KP; ++i) b[i] = (i < G) ? x[g + i] : -1.0f;
            sort_desc<KP>(b);
            merge_top_desc<KP>(run, b);
        }
    }
    __device__ __forceinline__ float theta(int K) const {
        float th = run[0];
#pragma unroll
        for (int i = 0; i < KP; ++i)
            if (i == K - 1) th = run[i];
        return th;
    }
    __device__ __forceinline__ int need(int K, float th) const {
        int gt = 0;
#pragma unroll
        for (int i = 0; i < KP; ++i)
            if (i < K && run[i] > th) ++gt;
        return K - gt;
    }
};

// Threshold pass over 4 consecutive scores: take everything above theta and the
// first `need` scores equal to theta; returns the 4 bits.
__device__ __forceinline__ uint32_t take4(float4 f, float th, int& need) {
    const float v[4] = {f.x, f.y, f.z, f.w};
    uint32_t w = 0u;
#pragma unroll
    for (int u = 0; u < 4; ++u) {
        const bool eq = v[u] == th;
        const bool take = (v[u] > th) || (eq && need > 0);
        need -= eq ? 1 : 0;
        w |= take ? (1u << u) : 0u;
    }
    return w;
}

// Top-K set of row[0..N) (N % 16 == 0, 1 <= K <= min(N, 32), values >= 0) as
// bits mask[e / 32] bit e % 32; mask must hold N / 32 rounded up words.
template <int KP>
__device__ __forceinline__ void row_topk_mask(const float* row, int N, int K, uint32_t* mask) {
    TopKAcc<KP> acc;
    acc.init();
    for (int c = 0; c < N; c += 16) {
        float x[16];
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const float4 f = __ldg(reinterpret_cast<const float4*>(row + c) + q);
            x[4 * q] = f.x;
            x[4 * q + 1] = f.y;
            x[4 * q + 2] = f.z;
            x[4 * q + 3] = f.w;
        }
        acc.add16(x);
    }
    const float th = acc.theta(K);
    // Every score >= theta: the Top-K set exactly when no more scores equal
    // theta than the set takes (the usual case), i.e. when it has K members.
    int cnt = 0;
    for (int c = 0; c < N; c += 32) {
        uint32_t w = 0u;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            if (c + 4 * q >= N) break;
            const float4 f = __ldg(reinterpret_cast<const float4*>(row + c) + q);
            w |= ((f.x >= th ? 1u : 0u) | (f.y >= th ? 2u : 0u) | (f.z >= th ? 4u : 0u) |
                  (f.w >= th ? 8u : 0u)) << (4 * q);
        }
        mask[c >> 5] = w;
        cnt += __popc(w);
    }
    if (cnt == K) return;
    // surplus scores equal to theta: take the lowest indices among them
    int need = acc.need(K, th);
    for (int c = 0; c < N; c += 32) {
        uint32_t w = 0u;
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            if (c + 4 * q >= N) break;
            w |= take4(__ldg(reinterpret_cast<const float4*>(row + c) + q), th, need) << (4 * q);
        }
        mask[c >> 5] = w;
    }
}

// Algorithm 2's pre-access refinement of the chain's cache with priorities
// a[e] + pS[e] (s^ST for the method, s^S for the Spatio-only ablation): the
// candidates A = Top_R of all experts in descending order, each skipped when
// resident, loaded into a free slot, or swapped for the lowest resident when
// strictly higher.  Returns the proactive loads.
//
// Only the non-resident members of A can change the cache, so they are taken
// one at a time in order -- the best remaining non-resident c -- and c is a
// member of A = Top_R exactly when fewer than R experts precede it in the
// order (its rank).  The first rank test is also the one that leaves the cache
// alone when the R first experts are all resident.  An original resident that
// a candidate evicted is never taken as a candidate itself: in the literal
// loop it would meet a cache whose lowest member is no lower than it and lose
// the strict test, ending the pass exactly as the rank test or the strict
// test ends it here.
//
// With nD_out, the first rank count also carries this lane's demand misses of
// `sel` against the cache as it stands; when that count ends the pass (the
// cache unchanged), *nD_out receives the warp's demand misses, else -1.
template <int V, bool ALL_VALID>
__device__ __forceinline__ int scan_refine(ChainRegs<V>& cr, const float (&pS)[V], uint32_t valid,
                                           int lane, int C, int R, uint32_t sel = 0u,
                                           int* nD_out = nullptr) {
    auto is_valid = [&](int v) { return ALL_VALID || ((valid >> v) & 1u); };
    uint32_t kS[V];
#pragma unroll
    for (int v = 0; v < V; ++v)
        kS[v] = is_valid(v) ? pkey(__fadd_rn(cr.aT[v], pS[v])) : 0u;
    uint32_t left = valid & ~cr.cache;         // non-residents not yet taken
    int pro = 0;
    if (nD_out) *nD_out = -1;
#pragma unroll 1
    for (int j = 0; j < R; ++j) {
        // the best remaining non-resident c: largest key, then lowest index
        uint32_t m[V];
#pragma unroll
        for (int v = 0; v < V; ++v) m[v] = ((left >> v) & 1u) ? kS[v] : 0u;
        uint32_t best = m[0];
#pragma unroll
        for (int v = 1; v < V; ++v) best = umax(best, m[v]);
        const uint32_t mx = __reduce_max_sync(kFull, best);
        if (mx == 0u) break;                   // no non-resident left
        // rank of c: experts with higher keys, and with equal keys at lower
        // indices (lanes before the owner; the owner's slots before c's).
        // Invalid slots hold key 0 and count for neither.  Fields of 9 bits
        // (counts <= N <= 256), the demand misses above them.
        uint32_t gt = 0u, eq = 0u;
#pragma unroll
        for (int v = 0; v < V; ++v) {
            gt += kS[v] > mx ? 1u : 0u;
            eq += kS[v] == mx ? 1u : 0u;
        }
        uint32_t packed = gt | (eq << 9);
        if (nD_out && j == 0) packed |= (uint32_t)__popc(sel & ~cr.cache) << 18;
        const uint32_t tot = __reduce_add_sync(kFull, packed);
        uint32_t rank = tot & 0x1ffu;
        const bool tie = ((tot >> 9) & 0x1ffu) > 1u;   // c shares its key
        int owner = 0;
        uint32_t cs = 0u;
        auto locate = [&]() {                  // c's lane and slot
            owner = __ffs(__ballot_sync(kFull, best == mx)) - 1;
#pragma unroll
            for (int v = V - 1; v >= 0; --v) cs = m[v] == mx ? (uint32_t)v : cs;   // lowest slot
        };
        if (tie) {                             // count those before c by index
            locate();
            const uint32_t c_slot = __shfl_sync(kFull, cs, owner);
            uint32_t before = 0u;
#pragma unroll
            for (int v = 0; v < V; ++v)
                before += (kS[v] == mx && (lane < owner || (lane == owner && (uint32_t)v < c_slot)))
                              ? 1u : 0u;
            rank += __reduce_add_sync(kFull, before);
        }
        if ((int)rank >= R) {                  // c is not among the top R, nor is any later one
            if (nD_out && j == 0) *nD_out = (int)(tot >> 18);
            break;
        }
        if (!tie) locate();
        const uint32_t cbit = (lane == owner) ? (1u << cs) : 0u;
        left &= ~cbit;
        if (cr.count < C) {                    // free slot: proactive load
            cr.cache |= cbit;
            ++cr.count;
            ++pro;
            continue;
        }
        uint32_t kv, vslot = 0u;
        const int vo = warp_last_member<V>(kS, cr.cache, lane, kv, vslot);
        if (mx > kv) {                         // strictly higher: replace the lowest resident
            const uint32_t vbit = (lane == vo) ? (1u << vslot) : 0u;
            cr.cache = (cr.cache & ~vbit) | cbit;
            ++pro;
        } else {
            break;                             // later candidates are no higher
        }
    }
    return pro;
}

// Refinement, access and UpdateCache of one access, given s^T = p^R + p^T,
// the Spatio prediction of the predecessor and the native Top-K set `sel`
// (this lane's V bits).  Updates the chain registers; returns the number of
// proactive loads and writes the demand misses to *n_miss.
template <int V, bool ALL_VALID>
__device__ __forceinline__ int scan_apply(ChainRegs<V>& cr, const float (&sT)[V],
                                          const float (&pS)[V], bool refine, uint32_t valid,
                                          int lane, int K, int C, int R, uint32_t sel,
                                          int* n_miss) {
    int nD_pre = -1;
    int pro = refine ? scan_refine<V, ALL_VALID>(cr, pS, valid, lane, C, R, sel, &nD_pre) : 0;

    // demand misses and UpdateCache (Algorithm 1)
    const uint32_t dem = sel & ~cr.cache;
    const int nD = nD_pre >= 0 ? nD_pre : (int)__reduce_add_sync(kFull, (uint32_t)__popc(dem));
    const int freeslots = C - cr.count;
    if (nD > freeslots) {
        uint32_t kT[V];
#pragma unroll
        for (int v = 0; v < V; ++v) kT[v] = pkey(sT[v]);
        uint32_t vset = cr.cache & ~sel;                       // V = C+ \ S
        for (int i = 0; i < nD - freeslots; ++i) {
            uint32_t kv, vslot = 0u;
            const int vo = warp_last_member<V>(kT, vset, lane, kv, vslot);
            const uint32_t rm = (lane == vo) ? (1u << vslot) : 0u;
            vset &= ~rm;
            cr.cache &= ~rm;
        }
        cr.count = C;
    } else {
        cr.count += nD;
    }
    cr.cache |= dem;
#pragma unroll
    for (int v = 0; v < V; ++v) cr.aT[v] = sT[v];
    cr.hits += (uint32_t)(K - nD);
    cr.misses += (uint32_t)nD;
    cr.pro += (uint32_t)pro;
    *n_miss = nD;
    return pro;
}

// This lane's cache bits as the chain's NW bitmask words at dst.
template <int V>
__device__ __forceinline__ void store_cache_words(uint32_t cache, int lane, int N, uint32_t* dst) {
    const int NW = (N + 31) >> 5;
    const int e0 = lane * V;
    for (int w = 0; w < NW; ++w) {
        const uint32_t contrib = (e0 < N && (e0 >> 5) == w) ? (cache << (e0 & 31)) : 0u;
        const uint32_t word = __reduce_or_sync(kFull, contrib);
        if (lane == 0) dst[w] = word;
    }
}

// One access at (t, l) from the three router probabilities: s^T, the native
// Top-K (given as a set, or popped in rank order when the trace wants the
// order), then scan_apply.  Writes the trace.
template <int V, bool ALL_VALID>
__device__ __forceinline__ void scan_step(ChainRegs<V>& cr, const float (&pR)[V],
                                          const float (&pT)[V], const float (&pS)[V],
                                          bool refine, uint32_t valid, int lane, int K, int C,
                                          int R, bool have_sel, uint32_t sel_in,
                                          uint8_t* topk_out, uint8_t* miss_out,
                                          uint8_t* pro_out, uint32_t* mid_out = nullptr,
                                          uint32_t* after_out = nullptr, int N = 0,
                                          uint32_t* sel_out = nullptr) {
    auto is_valid = [&](int v) { return ALL_VALID || ((valid >> v) & 1u); };
    float sT[V];
#pragma unroll
    for (int v = 0; v < V; ++v) sT[v] = __fadd_rn(pR[v], pT[v]);

    uint32_t sel = sel_in;
    int my_topk = 0;
    const bool want_topk = topk_out != nullptr;
    if (!have_sel) {
        KeyList<V> P;
#pragma unroll
        for (int v = 0; v < V; ++v) {
            P.k[v] = is_valid(v) ? pkey(pR[v]) : 0u;
            P.s[v] = v;
        }
        presort<V>(P);
        sel = 0u;
        for (int k = 0; k < K; ++k) {
            uint32_t kk, slot = 0u;
            const int owner = warp_pop_first<V>(P, lane, kk, slot);
            if (lane == owner) sel |= 1u << slot;
            if (want_topk) {
                const int e = __shfl_sync(kFull, lane * V + (int)slot, owner);
                if (lane == k) my_topk = e;
            }
        }
    }
    int nD, pro;
    if (mid_out) {
        // the refinement on its own, so the cache between the two phases is seen
        pro = refine ? scan_refine<V, ALL_VALID>(cr, pS, valid, lane, C, R) : 0;
        store_cache_words<V>(cr.cache, lane, N, mid_out);
        scan_apply<V, ALL_VALID>(cr, sT, pS, false, valid, lane, K, C, R, sel, &nD);
        cr.pro += (uint32_t)pro;
    } else {
        pro = scan_apply<V, ALL_VALID>(cr, sT, pS, refine, valid, lane, K, C, R, sel, &nD);
    }
    if (after_out) store_cache_words<V>(cr.cache, lane, N, after_out);
    if (sel_out) store_cache_words<V>(sel, lane, N, sel_out);
    if (want_topk && lane < K) topk_out[lane] = (uint8_t)my_topk;
    if (lane == 0) {
        if (miss_out) *miss_out = (uint8_t)nD;
        if (pro_out) *pro_out = (uint8_t)pro;
    }
}

// Bits of this lane's experts from the chain's bitmask words.
template <int V>
__device__ __forceinline__ uint32_t lane_bits(const uint32_t* words, int lane, int N) {
    const int e0 = lane * V;
    if (e0 >= N) return 0u;
    return (words[e0 >> 5] >> (e0 & 31)) & ((1u << V) - 1u);
}

// Warps (chains) per block of the stand-alone scans.  The scans are
// issue-bound with every chain resident at once, so their time is that of the
// most loaded SM: one-warp blocks spread the B*L chains within one warp per SM
// of even (3,072 chains over 152 SMs: 20 or 21 warps each, where blocks of
// four put 24 on some SMs and 20 on the rest).
constexpr int kScanWarps = 1;

// TRACED: compiled with the trace writes (any trace array given); the
// untraced kernel carries none of their code.
template <int V, bool ALL_VALID, int KP, bool TRACED>
__global__ void __launch_bounds__(32 * kScanWarps, (V >= 8 ? 12 : 24) / kScanWarps)
    cache_scan_kernel(ScanArgs a) {
    // Top-K sets of the next 32 tokens of each warp's chain, one row per token
    __shared__ uint32_t sel_s[kScanWarps][32][8];
    StateHeader* hdr = reinterpret_cast<StateHeader*>(a.state);
    const StateLayout lay = state_layout(a.B, a.L, a.N);
    ChainState* chains = reinterpret_cast<ChainState*>(a.state + lay.chains);
    float* retention = reinterpret_cast<float*>(a.state + lay.retention);
    float* carry = reinterpret_cast<float*>(a.state + lay.carry);

    const int lane = threadIdx.x & 31;
    const int chain = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const bool active = chain < a.B * a.L;

    const bool hdr_ok = hdr->magic == kStateMagic && hdr->L == a.L && hdr->N == a.N &&
                        hdr->K == a.K && hdr->C == a.C && hdr->R == a.R && hdr->B == a.B &&
                        hdr->policy == 0u;
    const int64_t t0 = hdr->t_next;
    const uint32_t parity = hdr->parity;

    uint32_t* err = &hdr->error;
    (void)err;                                  // read only by the checking build's bounds checks
    if (active && hdr_ok && CRC_IN_BOUNDS(a.trace_t0 >= 0 && a.trace_t0 + a.T <= a.trace_T, err)) {
        const int b = chain / a.L, l = chain % a.L;
        const int N = a.N, L = a.L, T = a.T;
        const size_t row = (size_t)3 * N;
        uint32_t valid = 0u;
#pragma unroll
        for (int v = 0; v < V; ++v)
            if (lane * V + v < N) valid |= 1u << v;
        const bool has = valid != 0u;

        ChainState& cs = chains[chain];
        ChainRegs<V> cr;
        cr.cache = lane_bits<V>(cs.bits, lane, N);
        cr.count = (int)__reduce_add_sync(kFull, (uint32_t)__popc(cr.cache));
        {
            Vec<V> x = load_vec<V>(retention + (size_t)chain * N + lane * V, has);
#pragma unroll
            for (int v = 0; v < V; ++v) cr.aT[v] = x.v[v];
        }
        cr.hits = cr.misses = cr.pro = 0u;

        const float* base = a.scores + lane * V;
        // debug builds: the unit a pointer is formed for lies inside scores [B][T][L]
        auto unit_ok = [&](int t, int ll) {
            return CRC_IN_BOUNDS(b < a.B && t >= 0 && t < T && ll >= 0 && ll < L, err);
        };
        auto unit_ptr = [&](int t, int ll) -> const float* {
            return base + (((size_t)b * T + t) * L + ll) * row;
        };
        const float* carry_in = carry + ((size_t)parity * a.B + b) * N + lane * V;
        auto pred_ptr = [&](int t) -> const float* {     // p^S of rho(t, l)
            if (l > 0) return unit_ptr(t, l - 1) + 2 * N;
            if (t > 0) return unit_ptr(t - 1, L - 1) + 2 * N;
            return carry_in;
        };
        const bool want_s = a.R > 0;

        // Without a trace only the Top-K *set* is needed: it does not depend on
        // the cache, so lane j computes it for token t + j ahead of the chain.
        const bool batch_sel = !TRACED || a.trace_topk == nullptr;
        uint32_t (*sel_rows)[8] = sel_s[(threadIdx.x >> 5) % kScanWarps];
        const float* row_base = a.scores + ((size_t)b * T * L + l) * row;   // token 0 of chain
        // running pointer to this lane's part of unit (b, t, l); p^S of rho(t, l)
        // sits at a fixed offset from it: unit (t, l-1), or (t-1, L-1) for l = 0
        const size_t tok = (size_t)L * row;
        const ptrdiff_t s_off = l > 0 ? (ptrdiff_t)2 * N - (ptrdiff_t)row
                                      : (ptrdiff_t)(L - 1) * (ptrdiff_t)row - (ptrdiff_t)tok +
                                            (ptrdiff_t)2 * N;
        const float* up = unit_ptr(0, l);

        Vec<V> cR = load_vec<V>(unit_ptr(0, l), has && unit_ok(0, l));
        Vec<V> cT = load_vec<V>(unit_ptr(0, l) + N, has && unit_ok(0, l));
        Vec<V> cS = load_vec<V>(pred_ptr(0), has && want_s && (t0 + 0 >= 1) &&
                                                 (l > 0 ? unit_ok(0, l - 1) : true));
        for (int t = 0; t < T; ++t) {
            if (batch_sel && (t & 31) == 0) {
                __syncwarp();
                if (t + lane < T && unit_ok(t + lane, l)) {
                    const float* r = row_base + (size_t)(t + lane) * L * row;
                    row_topk_mask<KP>(r, N, a.K, sel_rows[lane]);
                }
                __syncwarp();
            }
            uint32_t sel_in = 0u;
            if (batch_sel && has) {
                const uint32_t e0 = (uint32_t)lane * V;
                if (CRC_IN_BOUNDS((e0 >> 5) < 8u, err))
                    sel_in = (sel_rows[t & 31][e0 >> 5] >> (e0 & 31)) & ((1u << V) - 1u);
            }
            Vec<V> nR, nT, nS;
            if (t + 1 < T) {
                const bool ok1 = unit_ok(t + 1, l);
                const float* un = up + tok;
                nR = load_vec<V>(un, has && ok1);
                nT = load_vec<V>(un + N, has && ok1);
                nS = load_vec<V>(un + s_off, has && want_s &&
                                                 (l > 0 ? unit_ok(t + 1, l - 1) : unit_ok(t, L - 1)));
            }
            up += tok;
            const bool refine = want_s && (t0 + t >= 1);
            if constexpr (TRACED) {
                const size_t unit = ((size_t)b * a.trace_T + a.trace_t0 + t) * L + l;
                const size_t NWs = (size_t)((N + 31) >> 5);
                scan_step<V, ALL_VALID>(cr, cR.v, cT.v, cS.v, refine, valid, lane, a.K, a.C, a.R,
                                        batch_sel, sel_in,
                                        a.trace_topk ? a.trace_topk + unit * a.K : nullptr,
                                        a.trace_miss ? a.trace_miss + unit : nullptr,
                                        a.trace_pro ? a.trace_pro + unit : nullptr,
                                        a.trace_mid ? a.trace_mid + unit * NWs : nullptr,
                                        a.trace_after ? a.trace_after + unit * NWs : nullptr, N,
                                        a.trace_sel ? a.trace_sel + unit * NWs : nullptr);
            } else {                      // no trace: the set-valued Top-K, straight to the step
                float sT[V];
#pragma unroll
                for (int v = 0; v < V; ++v) sT[v] = __fadd_rn(cR.v[v], cT.v[v]);
                int nD;
                scan_apply<V, ALL_VALID>(cr, sT, cS.v, refine, valid, lane, a.K, a.C, a.R, sel_in,
                                         &nD);
            }
            // debug builds: every expert the step made resident lies in this
            // lane's range and the cache holds at most C experts
            (void)CRC_IN_BOUNDS((cr.cache & ~valid) == 0u && cr.count <= a.C, err);
            cR = nR;
            cT = nT;
            cS = nS;
        }

        // write back the chain
        const int NW = (N + 31) >> 5;
        for (int w = 0; w < NW; ++w) {
            const int e0 = lane * V;
            const uint32_t contrib = (has && (e0 >> 5) == w) ? (cr.cache << (e0 & 31)) : 0u;
            const uint32_t word = __reduce_or_sync(kFull, contrib);
            if (lane == 0) cs.bits[w] = word;
        }
        if (has && CRC_IN_BOUNDS(chain < a.B * a.L, err)) {
#pragma unroll
            for (int v = 0; v < V; ++v)
                if (lane * V + v < N) retention[(size_t)chain * N + lane * V + v] = cr.aT[v];
        }
        if (lane == 0) {
            cs.hits += cr.hits;
            cs.misses += cr.misses;
            cs.proactive += cr.pro;
        }
        // the last layer hands its final p^S to layer 0 of the next call
        if (l == L - 1 && has) {
            const float* src = unit_ptr(T - 1, L - 1) + 2 * N;
            float* dst = carry + ((size_t)(parity ^ 1u) * a.B + b) * N + lane * V;
#pragma unroll
            for (int v = 0; v < V; ++v)
                if (lane * V + v < N) dst[v] = src[v];
        }
    }

    // the last block to finish advances the token counter and flips the carry slot
    __syncthreads();
    if (threadIdx.x == 0) {
        if (!hdr_ok && blockIdx.x == 0) latch_error(&hdr->error, CRC_ESTATE);
        __threadfence();
        const uint32_t prev = atomicAdd(&hdr->done, 1u);
        if (prev == gridDim.x - 1) {
            __threadfence();
            if (hdr_ok) {
                hdr->t_next = t0 + a.T;
                hdr->parity = parity ^ 1u;
            }
            hdr->done = 0u;
            __threadfence();
        }
    }
}

}  // namespace crc
