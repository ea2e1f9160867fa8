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
// Reductions: order-preserving 32-bit keys of the fp32 scores reduced with
// redux.sync; ties resolved with a ballot (lowest lane = lowest index for an
// argmax, highest lane = highest index for the last-in-order argmin).
#pragma once

#include "crc_device.cuh"

namespace crc {

struct ScanArgs {
    const float* scores;     // [B][T][L][3][N]
    uint8_t* state;          // state buffer base
    uint8_t* trace_topk;     // [B][T][L][K] or null
    uint8_t* trace_miss;     // [B][T][L] or null
    uint8_t* trace_pro;      // [B][T][L] or null
    int trace_T, trace_t0;   // trace arrays span trace_T tokens; this call starts at trace_t0
    int B, T, L, N, K, C, R;
};

// Order-preserving key: larger float -> larger unsigned; -0 is mapped to +0.
// 0 is never produced for a non-NaN input and marks "no element".
__device__ __forceinline__ uint32_t okey(float x) {
    uint32_t u = __float_as_uint(x);
    u = (u == 0x80000000u) ? 0u : u;
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// First expert under (score desc, index asc) among eligible ones; -1 if none.
template <int V>
__device__ __forceinline__ int warp_argmax(const float (&s)[V], uint32_t elig, int lane,
                                           uint32_t& key) {
    uint32_t best = 0u;
    int bi = 0;
#pragma unroll
    for (int v = 0; v < V; ++v) {
        const uint32_t k = ((elig >> v) & 1u) ? okey(s[v]) : 0u;
        if (k > best) {
            best = k;
            bi = v;
        }
    }
    const uint32_t m = __reduce_max_sync(kFull, best);
    key = m;
    if (m == 0u) return -1;
    const uint32_t ball = __ballot_sync(kFull, best == m);
    const int src = __ffs(ball) - 1;
    return __shfl_sync(kFull, lane * V + bi, src);
}

// Last expert under (score desc, index asc) among eligible ones, i.e. the
// smallest score and, among equal scores, the highest index; -1 if none.
template <int V>
__device__ __forceinline__ int warp_argmin_last(const float (&s)[V], uint32_t elig, int lane,
                                                uint32_t& key) {
    uint32_t best = 0xffffffffu;
    int bi = -1;
#pragma unroll
    for (int v = 0; v < V; ++v) {
        if ((elig >> v) & 1u) {
            const uint32_t k = okey(s[v]);
            if (k <= best) {
                best = k;
                bi = v;
            }
        }
    }
    const uint32_t m = __reduce_min_sync(kFull, best);
    key = m;
    const uint32_t ball = __ballot_sync(kFull, bi >= 0 && best == m);
    if (ball == 0u) return -1;
    const int src = 31 - __clz(ball);
    return __shfl_sync(kFull, lane * V + bi, src);
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

// One access at (t, l).  Returns nothing; updates regs and writes the trace.
template <int V>
__device__ __forceinline__ void scan_step(ChainRegs<V>& cr, const float (&pR)[V],
                                          const float (&pT)[V], const float (&pS)[V],
                                          bool refine, uint32_t valid, int lane, int K, int C,
                                          int R, uint8_t* topk_out, uint8_t* miss_out,
                                          uint8_t* pro_out) {
    float sT[V];
#pragma unroll
    for (int v = 0; v < V; ++v) sT[v] = pR[v] + pT[v];

    int pro = 0;
    if (refine) {
        float sST[V];
#pragma unroll
        for (int v = 0; v < V; ++v) sST[v] = cr.aT[v] + pS[v];
        uint32_t taken = 0u;
        for (int r = 0; r < R; ++r) {
            uint32_t ke;
            const int e = warp_argmax<V>(sST, valid & ~taken, lane, ke);
            if (e < 0) break;
            const int owner = e / V;
            const uint32_t bit = 1u << (e % V);
            if (lane == owner) taken |= bit;
            const bool resident = __shfl_sync(kFull, (cr.cache & bit) != 0u, owner);
            if (resident) continue;
            if (cr.count < C) {                         // free slot: proactive load
                if (lane == owner) cr.cache |= bit;
                ++cr.count;
                ++pro;
                continue;
            }
            uint32_t kv;
            const int vic = warp_argmin_last<V>(sST, cr.cache, lane, kv);
            if (ke > kv) {                              // strictly higher: replace lowest
                if (lane == vic / V) cr.cache &= ~(1u << (vic % V));
                if (lane == owner) cr.cache |= bit;
                ++pro;
            } else {
                break;
            }
        }
    }

    // native Top-K
    uint32_t sel = 0u;
    int my_topk = 0;
    for (int k = 0; k < K; ++k) {
        uint32_t kk;
        const int e = warp_argmax<V>(pR, valid & ~sel, lane, kk);
        if (lane == e / V) sel |= 1u << (e % V);
        if (lane == k) my_topk = e;
    }

    // demand misses and UpdateCache (Algorithm 1)
    const uint32_t dem = sel & ~cr.cache;
    const int nD = (int)__reduce_add_sync(kFull, (uint32_t)__popc(dem));
    const int freeslots = C - cr.count;
    if (nD > freeslots) {
        uint32_t vset = cr.cache & ~sel;
        for (int i = 0; i < nD - freeslots; ++i) {
            uint32_t kv;
            const int vic = warp_argmin_last<V>(sT, vset, lane, kv);
            if (lane == vic / V) {
                vset &= ~(1u << (vic % V));
                cr.cache &= ~(1u << (vic % V));
            }
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

    if (topk_out && lane < K) topk_out[lane] = (uint8_t)my_topk;
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

template <int V>
__global__ void __launch_bounds__(128) cache_scan_kernel(ScanArgs a) {
    StateHeader* hdr = reinterpret_cast<StateHeader*>(a.state);
    const StateLayout lay = state_layout(a.B, a.L, a.N);
    ChainState* chains = reinterpret_cast<ChainState*>(a.state + lay.chains);
    float* retention = reinterpret_cast<float*>(a.state + lay.retention);
    float* carry = reinterpret_cast<float*>(a.state + lay.carry);

    const int lane = threadIdx.x & 31;
    const int chain = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const bool active = chain < a.B * a.L;

    const bool hdr_ok = hdr->magic == kStateMagic && hdr->L == a.L && hdr->N == a.N &&
                        hdr->K == a.K && hdr->C == a.C && hdr->R == a.R && hdr->B == a.B;
    const int64_t t0 = hdr->t_next;
    const uint32_t parity = hdr->parity;

    if (active && hdr_ok) {
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

        Vec<V> cR = load_vec<V>(unit_ptr(0, l), has);
        Vec<V> cT = load_vec<V>(unit_ptr(0, l) + N, has);
        Vec<V> cS = load_vec<V>(pred_ptr(0), has && want_s && (t0 + 0 >= 1));
        for (int t = 0; t < T; ++t) {
            Vec<V> nR, nT, nS;
            if (t + 1 < T) {
                nR = load_vec<V>(unit_ptr(t + 1, l), has);
                nT = load_vec<V>(unit_ptr(t + 1, l) + N, has);
                nS = load_vec<V>(pred_ptr(t + 1), has && want_s);
            }
            const size_t unit = ((size_t)b * a.trace_T + a.trace_t0 + t) * L + l;
            scan_step<V>(cr, cR.v, cT.v, cS.v, want_s && (t0 + t >= 1), valid, lane, a.K, a.C,
                         a.R, a.trace_topk ? a.trace_topk + unit * a.K : nullptr,
                         a.trace_miss ? a.trace_miss + unit : nullptr,
                         a.trace_pro ? a.trace_pro + unit : nullptr);
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
        if (has) {
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
