// Cache scans under the comparison policies of the paper's evaluation: the
// classical cache-update policies LRU, LFU and LRFU (lambda a multiple of
// 1/2; the paper uses 0.5) and the Spatio-only ablation (Algorithm 2's
// refinement on s^S = p^R_{t-1} + p^S_rho, LRU for demand misses; Sec. 4.3 and
// the appendix on ablations).  Same layout and reductions as the method's scan
// (cache_scan.cuh): one warp per (stream, layer) chain, lane i owns experts
// [iV, iV + V), priorities as ordered 32-bit keys.
//
// Readings (the paper names the policies and their references only):
//   - the classical policies only update the cache (no refinement, no
//     proactive load); each access demand-loads S \ C and, the cache being
//     full, evicts the member of C \ S with the lowest priority, ties to the
//     highest expert index, as Algorithm 1 does with s^T;
//   - LRU priority: the token of last use; LFU: the accesses that selected the
//     expert since it entered the cache; LRFU: CRF * F(t - t_last), the CRF
//     updated at each use to 1 + F(t - t_last) * CRF (1 on insertion), with
//     F(x) = 2^(-lambda x) computed in fp32 as 2^(-q) times fp32(2^(-1/2)) for
//     an odd number of halves, and 0 once q >= 126;
//   - Spatio-only: an expert its refinement loads counts as used at t.
#pragma once

#include "cache_scan.cuh"

namespace crc {

struct PolicyArgs {
    ScanArgs s;
    int policy;      // CRC_POLICY_*
    int lambda2;     // LRFU: lambda = lambda2 / 2
};

// F(dt) = 2^(-lambda dt) with lambda = lambda2 / 2.
__device__ __forceinline__ float lrfu_decay(int lambda2, uint32_t dt) {
    const uint32_t halves = (uint32_t)lambda2 * dt;
    const uint32_t q = halves >> 1;
    if (q >= 126u) return 0.f;
    float f = __uint_as_float((127u - q) << 23);                 // 2^-q, exact
    if (halves & 1u) f = __fmul_rn(f, 0.70710678118654752f);      // fp32(2^-1/2)
    return f;
}

// One access of the chain at token t under the policy POL (a CRC_POLICY_*
// value, fixed at compile time so that each policy's step carries only its
// own priority arithmetic).  aux: this lane's integer priorities (LRU,
// Spatio-only, LRFU: token of last use; LFU: count); cr.aT: the float ones
// (LRFU: CRF; Spatio-only: p^R of the previous token).
template <int V, bool ALL_VALID, int POL>
__device__ __forceinline__ void policy_step(ChainRegs<V>& cr, uint32_t (&aux)[V],
                                            const float (&pR)[V], const float (&pS)[V],
                                            bool refine, uint32_t valid, int lane,
                                            const PolicyArgs& a, uint32_t t, bool have_sel,
                                            uint32_t sel_in, uint8_t* topk_out,
                                            uint8_t* miss_out, uint8_t* pro_out) {
    auto is_valid = [&](int v) { return ALL_VALID || ((valid >> v) & 1u); };
    const int K = a.s.K, C = a.s.C;
    int pro = 0;
    if (POL == CRC_POLICY_SPATIO_LRU && refine) {
        const uint32_t before = cr.cache;
        pro = scan_refine<V, ALL_VALID>(cr, pS, valid, lane, C, a.s.R);
        const uint32_t loaded = cr.cache & ~before;
#pragma unroll
        for (int v = 0; v < V; ++v)
            if ((loaded >> v) & 1u) aux[v] = t;
    }
    // native Top-K on p^R: given as a set, or popped in rank order when the
    // trace wants the order
    uint32_t sel = sel_in;
    int my_topk = 0;
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
            if (topk_out) {
                const int e = __shfl_sync(kFull, lane * V + (int)slot, owner);
                if (lane == k) my_topk = e;
            }
        }
    }
    // demand loads; a full cache evicts the lowest priorities outside S (they
    // do not change while the access inserts, and inserted experts are in S)
    const uint32_t dem = sel & ~cr.cache;
    const uint32_t hit = sel & cr.cache;
    const int nD = (int)__reduce_add_sync(kFull, (uint32_t)__popc(dem));
    const int freeslots = C - cr.count;
    if (nD > freeslots) {
        uint32_t kV[V];
#pragma unroll
        for (int v = 0; v < V; ++v)
            kV[v] = POL == CRC_POLICY_LRFU
                        ? __float_as_uint(__fmul_rn(cr.aT[v], lrfu_decay(a.lambda2, t - aux[v])))
                        : aux[v];
        uint32_t vset = cr.cache & ~sel;
        for (int i = 0; i < nD - freeslots; ++i) {
            uint32_t kv, vslot = 0u;
            const int vo = warp_last_member<V>(kV, vset, lane, kv, vslot);
            const uint32_t rm = (lane == vo) ? (1u << vslot) : 0u;
            vset &= ~rm;
            cr.cache &= ~rm;
        }
        cr.count = C;
    } else {
        cr.count += nD;
    }
    cr.cache |= dem;
    // the selected experts' priorities after the access
#pragma unroll
    for (int v = 0; v < V; ++v) {
        if (!((sel >> v) & 1u)) continue;
        const bool h = (hit >> v) & 1u;
        if constexpr (POL == CRC_POLICY_LFU) {
            aux[v] = h ? aux[v] + 1u : 1u;
        } else if constexpr (POL == CRC_POLICY_LRFU) {
            cr.aT[v] = h ? __fadd_rn(1.f, __fmul_rn(lrfu_decay(a.lambda2, t - aux[v]), cr.aT[v]))
                         : 1.f;
            aux[v] = t;
        } else {
            aux[v] = t;
        }
    }
    if constexpr (POL == CRC_POLICY_SPATIO_LRU) {
#pragma unroll
        for (int v = 0; v < V; ++v) cr.aT[v] = pR[v];            // p^R_{t-1} for the next access
    }
    cr.hits += (uint32_t)(K - nD);
    cr.misses += (uint32_t)nD;
    cr.pro += (uint32_t)pro;
    if (topk_out && lane < K) topk_out[lane] = (uint8_t)my_topk;
    if (lane == 0) {
        if (miss_out) *miss_out = (uint8_t)nD;
        if (pro_out) *pro_out = (uint8_t)pro;
    }
}

template <int V, bool ALL_VALID, int KP, int POL>
__global__ void __launch_bounds__(32 * kScanWarps, (V >= 8 ? 12 : 24) / kScanWarps)
    cache_scan_policy_kernel(PolicyArgs pa) {
    // Top-K sets of the next 32 tokens of each warp's chain, one row per token
    __shared__ uint32_t sel_s[kScanWarps][32][8];
    const ScanArgs& a = pa.s;
    StateHeader* hdr = reinterpret_cast<StateHeader*>(a.state);
    const StateLayout lay = state_layout(a.B, a.L, a.N);
    ChainState* chains = reinterpret_cast<ChainState*>(a.state + lay.chains);
    float* val = reinterpret_cast<float*>(a.state + lay.retention);
    float* carry = reinterpret_cast<float*>(a.state + lay.carry);
    uint32_t* auxs = reinterpret_cast<uint32_t*>(a.state + lay.aux);

    const int lane = threadIdx.x & 31;
    const int chain = blockIdx.x * (blockDim.x >> 5) + (threadIdx.x >> 5);
    const bool active = chain < a.B * a.L;
    // a state belongs to one policy: the one that first used it
    const bool hdr_ok = hdr->magic == kStateMagic && hdr->L == a.L && hdr->N == a.N &&
                        hdr->K == a.K && hdr->C == a.C && hdr->R == a.R && hdr->B == a.B &&
                        (hdr->policy == (uint32_t)pa.policy || hdr->t_next == 0);
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
        uint32_t aux[V];
        {
            Vec<V> x = load_vec<V>(val + (size_t)chain * N + lane * V, has);
#pragma unroll
            for (int v = 0; v < V; ++v) {
                cr.aT[v] = x.v[v];
                aux[v] = (has && lane * V + v < N) ? auxs[(size_t)chain * N + lane * V + v] : 0u;
            }
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
        const bool want_s = POL == CRC_POLICY_SPATIO_LRU && a.R > 0;
        // without a rank-order trace the Top-K set is taken for 32 tokens at
        // a time, lane j for token t + j (it does not depend on the cache)
        const bool batch_sel = a.trace_topk == nullptr;
        uint32_t (*sel_rows)[8] = sel_s[(threadIdx.x >> 5) % kScanWarps];
        const float* row_base = a.scores + ((size_t)b * T * L + l) * row;   // token 0 of chain
        // running pointer to unit (b, t, l); p^S of rho(t, l) at a fixed offset
        const size_t tok = (size_t)L * row;
        const ptrdiff_t s_off = l > 0 ? (ptrdiff_t)2 * N - (ptrdiff_t)row
                                      : (ptrdiff_t)(L - 1) * (ptrdiff_t)row - (ptrdiff_t)tok +
                                            (ptrdiff_t)2 * N;
        const float* up = unit_ptr(0, l);
        const bool traced = a.trace_topk || a.trace_miss || a.trace_pro;

        Vec<V> cR = load_vec<V>(up, has);
        Vec<V> cS = load_vec<V>(pred_ptr(0), has && want_s && t0 >= 1);
        for (int t = 0; t < T; ++t) {
            if (batch_sel && (t & 31) == 0) {
                __syncwarp();
                if (t + lane < T)
                    row_topk_mask<KP>(row_base + (size_t)(t + lane) * tok, N, a.K, sel_rows[lane]);
                __syncwarp();
            }
            uint32_t sel_in = 0u;
            if (batch_sel && has) {
                const uint32_t e0 = (uint32_t)lane * V;
                sel_in = (sel_rows[t & 31][e0 >> 5] >> (e0 & 31)) & ((1u << V) - 1u);
            }
            Vec<V> nR, nS;
            if (t + 1 < T) {
                nR = load_vec<V>(up + tok, has);
                nS = load_vec<V>(up + tok + s_off, has && want_s);
            }
            up += tok;
            const bool refine = want_s && (t0 + t >= 1);
            if (traced) {
                const size_t unit = ((size_t)b * a.trace_T + a.trace_t0 + t) * L + l;
                policy_step<V, ALL_VALID, POL>(cr, aux, cR.v, cS.v, refine, valid, lane, pa,
                                               (uint32_t)(t0 + t), batch_sel, sel_in,
                                          a.trace_topk ? a.trace_topk + unit * a.K : nullptr,
                                          a.trace_miss ? a.trace_miss + unit : nullptr,
                                          a.trace_pro ? a.trace_pro + unit : nullptr);
            } else {
                policy_step<V, ALL_VALID, POL>(cr, aux, cR.v, cS.v, refine, valid, lane, pa,
                                               (uint32_t)(t0 + t), true, sel_in, nullptr,
                                               nullptr, nullptr);
            }
            cR = nR;
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
                if (lane * V + v < N) {
                    val[(size_t)chain * N + lane * V + v] = cr.aT[v];
                    auxs[(size_t)chain * N + lane * V + v] = aux[v];
                }
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

    // the last block to finish advances the token counter, flips the carry
    // slot and records the policy
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
                hdr->policy = (uint32_t)pa.policy;
            }
            hdr->done = 0u;
            __threadfence();
        }
    }
}

}  // namespace crc
