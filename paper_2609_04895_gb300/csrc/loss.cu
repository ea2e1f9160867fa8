// Soft Top-B cache-coverage losses and their gradient (Sec. 3.1-3.4), from the
// router probabilities: one warp per (stream, layer, token chunk), or for
// short rows (N = 16, 32 with top_b <= 16) one or two lanes per such task.
//
// For a priority s over N experts and a target distribution q:
//   theta_B(s) = the B-th largest entry of s,
//   m_e        = sigmoid((s_e - theta_B(s)) / tau),
//   l(s, q)    = sum_e q_e (1 - m_e).
// Step t of layer l evaluates two terms that share their inputs:
//   l^T_{t,l}    = l(s^T_{t,l}, p^R_{t+1,l}),            s^T = p^R + p^T   (Sec. 3.2)
//   l^ST_{t+1,l} = l(s^T_{t,l} + p^S_{rho(t+1,l)}, p^R_{t+1,l})            (Sec. 3.3)
// (a^T_{t+1,l} = s^T_{t,l}, and both targets are p^R_{t+1,l}).  With
// g = dl/ds (through s_e and through theta_B, whose subgradient goes to the
// element at position B of the order score descending, index ascending) and
// gq = dl/dq = 1 - m, the gradient of w_T L_T + w_ST L_ST (means over the valid
// positions, cT = w_T / |Omega_T|, cST = w_ST / |Omega_ST|) with respect to the
// probabilities is
//   dp^R_{t,l}          = cT gT_t + cST gST_{t+1} + cT gqT_{t-1} + cST gqST_t
//   dp^T_{t,l}          = cT gT_t + cST gST_{t+1}
//   dp^S_{rho(t+1,l)}   = cST gST_{t+1}
// since the native distributions are differentiable both as priorities and as
// targets (Sec. 3.4).  Every one of these rows is complete once the warp of
// layer l has finished step t -- the p^S row of rho(t+1,l) receives from
// l^ST_{t+1,l} alone -- so the warp applies each head's softmax backward,
// dz = p (dp - <p, dp>), and stores the row at once: every probability row is
// read once, every gradient row written once, and nothing is accumulated
// across warps.  A chunk that does not start at token 0 first evaluates the
// two terms of the token before it (the halo) for the target part of its
// first p^R row.
//
// Arithmetic: s^T and s^ST are formed by the same fp32 additions as the cache
// scan, so theta_B and the element carrying its subgradient are exact
// decisions on fp32 values; the sigmoid and everything after it are fp32
// (exp(-|x|) with the hardware exponential), the per-task loss sums fp64.
#include <cuda_runtime.h>
#include <stdint.h>

#include <atomic>

#include "cache_scan.cuh"
#include "crc_internal.h"

namespace crc {
namespace {

constexpr int kLossWarps = 8;

struct LossArgs {
    const float* probs;   // [B][T][L][3][N]
    float* loss;          // [B][T][L][2] (l^T, l^ST) or null
    float* grad;          // [B][T][L][3][N] or null
    double* partial;      // [tasks][2] per-task sums of l^T and l^ST, or null
    int B, T, L, N, heads, top_b, chunk, nchunks;
    float k2;             // log2(e) / tau
    float cT, cST;        // w_T / |Omega_T|, w_ST / |Omega_ST|: coefficients of dl/dq
    float gT, gST;        // the same over tau: coefficients of -w (dl/ds = -w / tau)
};

// Row element e = V * lane + j lives in slot j of `lane` (lanes >= N / V idle).
template <int V>
__device__ __forceinline__ void load_row(float (&x)[V], const float* row, int lane, bool valid) {
    if (!valid) {
#pragma unroll
        for (int j = 0; j < V; ++j) x[j] = 0.f;
        return;
    }
    const float* p = row + V * lane;
    if constexpr (V == 1) {
        x[0] = __ldcs(p);
    } else if constexpr (V == 2) {
        const float2 v = __ldcs(reinterpret_cast<const float2*>(p));
        x[0] = v.x;
        x[1] = v.y;
    } else {
#pragma unroll
        for (int i = 0; i < V; i += 4) {
            const float4 v = __ldcs(reinterpret_cast<const float4*>(p + i));
            x[i] = v.x;
            x[i + 1] = v.y;
            x[i + 2] = v.z;
            x[i + 3] = v.w;
        }
    }
}

template <int V>
__device__ __forceinline__ void store_row(float* row, const float (&x)[V], int lane, bool valid) {
    if (!valid) return;
    float* p = row + V * lane;
    if constexpr (V == 1) {
        __stcs(p, x[0]);
    } else if constexpr (V == 2) {
        __stcs(reinterpret_cast<float2*>(p), make_float2(x[0], x[1]));
    } else {
#pragma unroll
        for (int i = 0; i < V; i += 4)
            __stcs(reinterpret_cast<float4*>(p + i), make_float4(x[i], x[i + 1], x[i + 2], x[i + 3]));
    }
}

// Bit pattern of theta_B(s).  The entries are >= 0, so their bit patterns
// order like their values; the search fixes the bits of the largest probe x
// with #{k >= x} >= B from the most significant bit down, starting below the
// bits all valid keys share, and stops early once exactly B keys are >= x
// (theta is then the least of them).  Idle lanes hold key 0 and every probe
// is >= 1, so they are never counted.
template <int V>
__device__ __forceinline__ uint32_t theta_key(const uint32_t (&k)[V], bool valid, int top_b) {
    uint32_t lo = 0xffffffffu, hi = 0u;
#pragma unroll
    for (int j = 0; j < V; ++j) {
        lo &= valid ? k[j] : 0xffffffffu;
        hi |= k[j];
    }
    lo = __reduce_and_sync(kFull, lo);
    hi = __reduce_or_sync(kFull, hi);
    const uint32_t diff = lo ^ hi;
    if (diff == 0u) return lo;                      // all valid keys equal
    int bit = 31 - __clz(diff);
    uint32_t prefix = lo & ~((2u << bit) - 1u);     // the shared high bits
    const uint32_t need = (uint32_t)top_b;
#pragma unroll 1
    for (; bit >= 0; --bit) {
        const uint32_t x = prefix | (1u << bit);
        uint32_t c = 0;
#pragma unroll
        for (int j = 0; j < V; ++j) c += k[j] >= x ? 1u : 0u;
        const uint32_t n = __reduce_add_sync(kFull, c);
        if (n >= need) {
            prefix = x;
            if (n == need) {
                uint32_t m = 0xffffffffu;
#pragma unroll
                for (int j = 0; j < V; ++j) m = k[j] >= x && k[j] < m ? k[j] : m;
                return __reduce_min_sync(kFull, m);
            }
        }
    }
    return prefix;
}

// theta_B from a guess g (the same term's theta at the previous token, which
// is close: consecutive tokens route alike).  With n = #{k >= g}, theta is
// the (n - B + 1)-th smallest key >= g, or the (B - n)-th largest key < g;
// those are taken one distinct value at a time (redux min / max, then the
// count of that value, so ties count with their multiplicity).  More than
// kExtract rounds, or a round without a candidate, falls back to the bit
// search.  Exact either way.
constexpr int kExtract = 6;

template <int V>
__device__ __forceinline__ uint32_t theta_near(const uint32_t (&k)[V], bool valid, int top_b,
                                               uint32_t g) {
    uint32_t c = 0;
#pragma unroll
    for (int j = 0; j < V; ++j) c += valid && k[j] >= g ? 1u : 0u;
    const int n = (int)__reduce_add_sync(kFull, c);
    if (n >= top_b) {
        int r = n - top_b;                          // keys >= g that rank below theta
        uint32_t lower = g;
        if (r < kExtract) {
#pragma unroll 1
            for (int it = 0; it < kExtract; ++it) {
                uint32_t m = 0xffffffffu;
#pragma unroll
                for (int j = 0; j < V; ++j) m = valid && k[j] >= lower && k[j] < m ? k[j] : m;
                m = __reduce_min_sync(kFull, m);
                uint32_t e = 0;
#pragma unroll
                for (int j = 0; j < V; ++j) e += valid && k[j] == m ? 1u : 0u;
                const int ce = (int)__reduce_add_sync(kFull, e);
                if (ce == 0) break;                 // no key left (m is the sentinel)
                if (ce > r) return m;
                r -= ce;
                lower = m + 1u;
            }
        }
    } else {
        int need = top_b - n;                       // theta is the need-th largest key < g
        uint32_t upper = g;
        if (need <= kExtract) {
#pragma unroll 1
            for (int it = 0; it < kExtract; ++it) {
                uint32_t m = 0u;
#pragma unroll
                for (int j = 0; j < V; ++j) m = valid && k[j] < upper && k[j] > m ? k[j] : m;
                m = __reduce_max_sync(kFull, m);
                uint32_t e = 0;
#pragma unroll
                for (int j = 0; j < V; ++j) e += valid && k[j] < upper && k[j] == m ? 1u : 0u;
                const int ce = (int)__reduce_add_sync(kFull, e);
                if (ce == 0) break;                 // no key below `upper`
                if (ce >= need) return m;
                need -= ce;
                upper = m;
            }
        }
    }
    return theta_key<V>(k, valid, top_b);
}

// Slot of this lane holding the element at position B of the total order
// (score descending, index ascending), or -1: the keys above theta come
// first, then the keys equal to theta by ascending index V * lane + j.
template <int V>
__device__ __forceinline__ int theta_slot(const uint32_t (&k)[V], bool valid, uint32_t th,
                                          int top_b, int lane) {
    uint32_t gt = 0, eq = 0;
#pragma unroll
    for (int j = 0; j < V; ++j) {
        gt += k[j] > th ? 1u : 0u;
        eq += valid && k[j] == th ? 1u : 0u;
    }
    const uint32_t both = __reduce_add_sync(kFull, gt | (eq << 16));   // counts <= 256 each
    const int rank = top_b - (int)(both & 0xffffu);                    // 1-based among the ties
    int before = 0;
    if ((both >> 16) > 1u) {                        // ties at theta: exclusive scan of eq
        uint32_t inc = eq;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t y = __shfl_up_sync(kFull, inc, o);
            if (lane >= o) inc += y;
        }
        before = (int)(inc - eq);
    }
    int slot = -1, seen = before;
#pragma unroll
    for (int j = 0; j < V; ++j)
        if (valid && k[j] == th && ++seen == rank) slot = j;
    return slot;
}

__device__ __forceinline__ float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

__device__ __forceinline__ float rcp_approx(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// One coverage term before its reductions.  With d = s_e - theta_B and
// u = sigmoid(|d| / tau), v = 1 - u: om_e = 1 - m_e (v if d >= 0, else u) and
// w_e = q_e m_e (1 - m_e) = q_e u v, so that dl/ds_e = (W [e = e*] - w_e) / tau
// with W = sum_e w_e (the second part through theta_B = s_{e*}).  Adds the
// lane's share of l and of W to loss and wsum; the slot of e* comes back.
template <int V>
__device__ __forceinline__ int coverage(const float (&s)[V], const float (&q)[V], bool valid,
                                        int top_b, float k2, int lane, uint32_t& guess,
                                        float (&w)[V], float (&om)[V], float& loss, float& wsum) {
    uint32_t k[V];
#pragma unroll
    for (int j = 0; j < V; ++j) k[j] = valid ? __float_as_uint(s[j]) : 0u;
    const uint32_t th = theta_near<V>(k, valid, top_b, guess);
    guess = th;
    const int js = theta_slot<V>(k, valid, th, top_b, lane);
    const float theta = __uint_as_float(th);
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const float d = s[j] - theta;
        const float E = ex2_approx(-fabsf(d) * k2);     // exp(-|d| / tau), in (0, 1]
        const float u = rcp_approx(1.f + E);
        const float v = E * u;
        om[j] = d >= 0.f ? v : u;
        loss = fmaf(q[j], om[j], loss);
        w[j] = q[j] * (u * v);
        wsum += w[j];
    }
    return js;
}

// Sums of four per-lane values over the warp in one transposing butterfly
// (6 shuffles): lanes 0-7 end with the sum of a, 8-15 of b, 16-23 of c,
// 24-31 of d.
__device__ __forceinline__ float warp_sum4(float a, float b, float c, float d, int lane) {
    const bool h16 = (lane & 16) != 0;
    const float x0 = (h16 ? c : a) + __shfl_xor_sync(kFull, h16 ? a : c, 16);
    const float x1 = (h16 ? d : b) + __shfl_xor_sync(kFull, h16 ? b : d, 16);
    const bool h8 = (lane & 8) != 0;
    float y = (h8 ? x1 : x0) + __shfl_xor_sync(kFull, h8 ? x0 : x1, 8);
    y += __shfl_xor_sync(kFull, y, 4);
    y += __shfl_xor_sync(kFull, y, 2);
    y += __shfl_xor_sync(kFull, y, 1);
    return y;
}

template <int V>
__device__ __forceinline__ void store_zero(float* row, int lane, bool valid) {
    float z[V];
#pragma unroll
    for (int j = 0; j < V; ++j) z[j] = 0.f;
    store_row<V>(row, z, lane, valid);
}

// Softmax backward of up to three head rows and their stores:
// dz = p (dp - <p, dp>), the three inner products in one butterfly.
template <int V>
__device__ __forceinline__ void store_dz3(float* rR, float* rT, float* rS, const float (&pR)[V],
                                          const float (&dR)[V], const float (&pT)[V],
                                          const float (&dT)[V], const float (&pS)[V],
                                          const float (&dS)[V], bool with_s, int lane,
                                          bool valid) {
    float a = 0.f, b = 0.f, c = 0.f;
#pragma unroll
    for (int j = 0; j < V; ++j) {
        a = fmaf(pR[j], dR[j], a);
        b = fmaf(pT[j], dT[j], b);
        c = fmaf(pS[j], dS[j], c);
    }
    const float y = warp_sum4(a, b, c, 0.f, lane);
    const float dotR = __shfl_sync(kFull, y, 0);
    const float dotT = __shfl_sync(kFull, y, 8);
    const float dotS = __shfl_sync(kFull, y, 16);
    float o[V];
#pragma unroll
    for (int j = 0; j < V; ++j) o[j] = pR[j] * (dR[j] - dotR);
    store_row<V>(rR, o, lane, valid);
#pragma unroll
    for (int j = 0; j < V; ++j) o[j] = pT[j] * (dT[j] - dotT);
    store_row<V>(rT, o, lane, valid);
    if (with_s) {
#pragma unroll
        for (int j = 0; j < V; ++j) o[j] = pS[j] * (dS[j] - dotS);
        store_row<V>(rS, o, lane, valid);
    }
}

// Both terms of step t of layer l from s^T = p^R_t + p^T_t, p^S_{rho(t+1,l)}
// and the target q = p^R_{t+1}: their losses (lane 0: l^T, lane 16: l^ST in
// the returned value), gT = tau dl^T/ds, gST likewise, and the target parts.
template <int V>
__device__ __forceinline__ float step_terms(const float (&pR)[V], const float (&pT)[V],
                                            const float (&pS)[V], const float (&q)[V],
                                            bool st, bool valid, int top_b, float k2, int lane,
                                            uint32_t (&guess)[2], float (&wT)[V], float (&omT)[V],
                                            float (&wST)[V], float (&omST)[V]) {
    float s[V];
#pragma unroll
    for (int j = 0; j < V; ++j) s[j] = __fadd_rn(pR[j], pT[j]);
    float lT = 0.f, sT = 0.f, lST = 0.f, sST = 0.f;
    const int jT = coverage<V>(s, q, valid, top_b, k2, lane, guess[0], wT, omT, lT, sT);
    int jST = -1;
    if (st) {
#pragma unroll
        for (int j = 0; j < V; ++j) s[j] = __fadd_rn(s[j], pS[j]);
        jST = coverage<V>(s, q, valid, top_b, k2, lane, guess[1], wST, omST, lST, sST);
    }
    const float y = warp_sum4(lT, sT, lST, sST, lane);
    const float WT = __shfl_sync(kFull, y, 8);
    const float WST = __shfl_sync(kFull, y, 24);
    // w <- w - W [e = e*], so that dl/ds = -w / tau
#pragma unroll
    for (int j = 0; j < V; ++j) {
        if (j == jT) wT[j] -= WT;
        if (j == jST) wST[j] -= WST;
    }
    return y;
}

// Resident blocks per SM.  With one element per lane (N <= 32) a step is a
// chain of warp-wide reductions over short rows and the kernel is latency-
// bound: 8 blocks (64 warps, 32 registers, a few spilled) run the GPT-OSS-shaped
// workload in 2.20 ms against 2.66 ms with 4 blocks (56 registers).
template <int V>
constexpr int loss_blocks() { return V >= 8 ? 2 : (V == 1 ? 8 : 4); }

// ST: the Spatio term too (heads = 3), fixed at compile time.
template <int V, bool ALL_VALID, bool ST>
__global__ void __launch_bounds__(32 * kLossWarps, loss_blocks<V>()) cache_loss_kernel(const LossArgs a) {
    const int lane = threadIdx.x & 31;
    const int task = blockIdx.x * kLossWarps + (threadIdx.x >> 5);
    if (task >= a.B * a.L * a.nchunks) return;
    const int T = a.T, L = a.L, N = a.N;
    const int l = task % L;
    const int c = (task / L) % a.nchunks;
    const int b = task / (L * a.nchunks);
    const int t0 = c * a.chunk;
    const int t1 = min(T, t0 + a.chunk);
    const bool valid = ALL_VALID || lane < N / V;
    constexpr bool st = ST;
    const bool want_grad = a.grad != nullptr;
    const float k2 = a.k2, cT = a.cT, cST = a.cST, gT = a.gT, gST = a.gST;
    const size_t row3 = (size_t)3 * N;
    const size_t tok = (size_t)L * row3;                      // one token of one stream
    // row pointers at token t of unit (b, t, l) (load_row / store_row add the
    // lane's V elements); p^S of rho(t + 1, l) is (t, L - 1) for l = 0 and
    // (t + 1, l - 1) otherwise
    const size_t base = ((size_t)b * T * L + l) * row3;
    const size_t s_off = l > 0 ? tok + (size_t)2 * N - row3 : (size_t)(L - 1 - l) * row3 + 2 * N;
    const float* pp = a.probs + base + (size_t)t0 * tok;
    float* gp = want_grad ? a.grad + base + (size_t)t0 * tok : nullptr;
    float* lossp = a.loss ? a.loss + (((size_t)b * T + t0) * L + l) * 2 : nullptr;

    float pR[V], pT[V], q[V], pS[V], carry[V];
    float wT[V], omT[V], wST[V], omST[V];
#pragma unroll
    for (int j = 0; j < V; ++j) {
        carry[j] = 0.f;
        wST[j] = omST[j] = pS[j] = 0.f;
    }
    double sumT = 0.0, sumST = 0.0;
    uint32_t guess[2] = {0u, 0u};                             // theta^T, theta^ST of the last step

    if (t0 > 0) {
        // halo: the two terms of step t0 - 1 give the target part of p^R_{t0}
        const float* hp = pp - tok;
        load_row<V>(pR, hp, lane, valid);
        load_row<V>(pT, hp + N, lane, valid);
        load_row<V>(q, pp, lane, valid);
        if (st) load_row<V>(pS, hp + s_off, lane, valid);
        step_terms<V>(pR, pT, pS, q, st, valid, a.top_b, k2, lane, guess, wT, omT, wST, omST);
#pragma unroll
        for (int j = 0; j < V; ++j) {
            carry[j] = fmaf(cT, omT[j], cST * omST[j]);
            pR[j] = q[j];
        }
    } else {
        load_row<V>(pR, pp, lane, valid);
        if (lossp && lane == 0) lossp[1] = 0.f;                   // no l^ST at t = 0
        if (st && want_grad && l > 0) store_zero<V>(gp + 2 * N - row3, lane, valid);
    }

#pragma unroll 1
    for (int t = t0; t < t1; ++t, pp += tok) {
        load_row<V>(pT, pp + N, lane, valid);
        float dR[V], dT[V], dS[V];
        const bool next = t + 1 < T;
        if (next) {
            load_row<V>(q, pp + tok, lane, valid);
            if (st) load_row<V>(pS, pp + s_off, lane, valid);
            const float y = step_terms<V>(pR, pT, pS, q, st, valid, a.top_b, k2, lane, guess, wT,
                                          omT, wST, omST);
            if (lane == 0) {
                sumT += (double)y;
                if (lossp) lossp[0] = y;
            } else if (lane == 16) {
                sumST += (double)y;
                if (lossp) lossp[(size_t)L * 2 + 1] = st ? y : 0.f;
            }
#pragma unroll
            for (int j = 0; j < V; ++j) {
                const float gs = -fmaf(gT, wT[j], gST * wST[j]);
                dT[j] = gs;
                dR[j] = carry[j] + gs;
                dS[j] = -gST * wST[j];
                carry[j] = fmaf(cT, omT[j], cST * omST[j]);
            }
        } else {
            // last token: no l^T here, no l^ST after it
            if (lossp && lane == 0) lossp[0] = 0.f;
#pragma unroll
            for (int j = 0; j < V; ++j) {
                dR[j] = carry[j];
                dT[j] = dS[j] = 0.f;
            }
            if (st && want_grad && l == 0) store_zero<V>(gp + s_off, lane, valid);
        }
        if (want_grad) {
            store_dz3<V>(gp, gp + N, gp + s_off, pR, dR, pT, dT, pS, dS, st && next, lane,
                         valid);
            gp += tok;
        }
        if (lossp) lossp += (size_t)L * 2;
#pragma unroll
        for (int j = 0; j < V; ++j) pR[j] = q[j];
    }
    if (a.partial) {
        sumT = __shfl_sync(kFull, sumT, 0);
        sumST = __shfl_sync(kFull, sumST, 16);
        if (lane == 0) {
            a.partial[(size_t)task * 2 + 0] = sumT;
            a.partial[(size_t)task * 2 + 1] = sumST;
        }
    }
}

// ---------------------------------------------------------------------------
// Short rows (N = 16 or 32, top_b <= 16).  One warp-wide reduction per row
// quantity leaves such rows latency- and issue-bound, so here a row is held
// by NL = N / 16 lanes, 16 elements each, a warp runs 32 / NL tasks side by
// side, and every per-row quantity is lane-serial work plus at most one
// exchange with the partner lane (shuffle xor 1).  theta_B is the top_b-th
// entry of the running top KP (sorting networks over the lane's 16 values,
// merged with the partner's), e* the need-th value equal to it in index
// order; per element the arithmetic is that of the warp-per-row kernel.
// ---------------------------------------------------------------------------
constexpr int kRowE = 16;       // row elements per lane
constexpr int kRowWarps = 4;    // warps per block of the short-row kernel

template <int NL>
__device__ __forceinline__ float pair_sum(float x) {
    if constexpr (NL == 2) x += __shfl_xor_sync(kFull, x, 1);
    return x;
}

__device__ __forceinline__ void load16(float (&x)[kRowE], const float* p, bool ok) {
    if (!ok) {
#pragma unroll
        for (int j = 0; j < kRowE; ++j) x[j] = 0.f;
        return;
    }
#pragma unroll
    for (int i = 0; i < kRowE / 4; ++i) {
        const float4 v = __ldcs(reinterpret_cast<const float4*>(p) + i);
        x[4 * i] = v.x;
        x[4 * i + 1] = v.y;
        x[4 * i + 2] = v.z;
        x[4 * i + 3] = v.w;
    }
}

__device__ __forceinline__ void store16(float* p, const float (&x)[kRowE]) {
#pragma unroll
    for (int i = 0; i < kRowE / 4; ++i)
        __stcs(reinterpret_cast<float4*>(p) + i,
               make_float4(x[4 * i], x[4 * i + 1], x[4 * i + 2], x[4 * i + 3]));
}

// 16-byte asynchronous copy global -> shared (zero-filled when !ok; the
// address is then not read), and its group fences.
__device__ __forceinline__ void cp_async16(float4* smem, const float* gmem, bool ok) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(smem_u32(smem)),
                 "l"(gmem), "r"(ok ? 16 : 0)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}
__device__ __forceinline__ void cp_async_wait1() {
    asm volatile("cp.async.wait_group 1;" ::: "memory");
}

// theta_B of the row (the same in both lanes of a pair) and, in `slot`, this
// lane's slot holding e*, the element at position top_b of the order (score
// descending, index ascending), or -1.  The lower lane of a pair holds
// elements 0-15, the upper 16-31.
template <int NL, int KP>
__device__ __forceinline__ float row_theta(const float (&s)[kRowE], int top_b, int half, int lane,
                                           int& slot) {
    // the lane's top KP, descending: sort the groups of KP values, merge them
    float run[KP];
#pragma unroll
    for (int i = 0; i < KP; ++i) run[i] = s[i];
    sort_desc<KP>(run);
#pragma unroll
    for (int g = KP; g < kRowE; g += KP) {
        float b[KP];
#pragma unroll
        for (int i = 0; i < KP; ++i) b[i] = s[g + i];
        sort_desc<KP>(b);
        merge_top_desc<KP>(run, b);
    }
    if constexpr (NL == 2) {                    // and the partner lane's
        float o[KP];
#pragma unroll
        for (int i = 0; i < KP; ++i) o[i] = __shfl_xor_sync(kFull, run[i], 1);
        merge_top_desc<KP>(run, o);
    }
    float th = run[0];
#pragma unroll
    for (int i = 1; i < KP; ++i) th = i == top_b - 1 ? run[i] : th;
    int above = 0;                              // entries above theta, all within the top KP
#pragma unroll
    for (int i = 0; i < KP; ++i) above += (i < top_b && run[i] > th) ? 1 : 0;
    // e* is the (top_b - above)-th entry equal to theta in index order
    uint32_t eq = 0u;
#pragma unroll
    for (int j = 0; j < kRowE; ++j) eq |= s[j] == th ? 1u << j : 0u;
    int r = top_b - above;
    if constexpr (NL == 2) {
        const int eq_lo = __popc(__shfl_sync(kFull, eq, lane & ~1));
        if (half) r -= eq_lo;
    }
    slot = (r >= 1 && r <= __popc(eq)) ? (int)__fns(eq, 0u, r) : -1;
    return th;
}

// Rows of one step in shared memory: float4 i of thread x at st[i][x];
// quads 0-3 p^T_t, 4-7 p^R_{t+1}, 8-11 p^S_{rho(t+1)} (16 elements each).
using RowStage = float4[12][32 * kRowWarps];

// One 16-byte shared-memory load, issued where it is written: kept whole
// (a warp's loads of a quad are then contiguous) and ordered after the
// cp.async wait.
__device__ __forceinline__ float4 lds4(const float4& p) {
    float4 v;
    asm volatile("ld.shared.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(smem_u32(&p)));
    return v;
}

__device__ __forceinline__ float f4(const float4& v, int c) {
    return c == 0 ? v.x : c == 1 ? v.y : c == 2 ? v.z : v.w;
}

// One step's two terms from p^R_t (registers), p^T_t, p^S_{rho(t+1)} and the
// target q = p^R_{t+1} (the stage): returns (l^T, l^ST); dT = dl/dp^T,
// dR = carry + dT (carry: the target part of p^R_t from the step before),
// dS = dl/dp^S, all scaled by the objective's coefficients; carry becomes the
// target part of p^R_{t+1}.  s^T and s^ST are re-formed where they are used,
// by the same fp32 additions, so they need no registers across the step.
template <int NL, int KP>
__device__ __forceinline__ float2 rows_step(const float (&pR)[kRowE], const RowStage& sg, int x,
                                            bool st, int top_b, const LossArgs& a, int half,
                                            int lane, float (&carry)[kRowE], float (&dR)[kRowE],
                                            float (&dT)[kRowE], float (&dS)[kRowE]) {
    int jT, jST = -1;
    float thT, thST = 0.f;
    {
        float s[kRowE];
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float4 f = lds4(sg[i][x]);
#pragma unroll
            for (int c = 0; c < 4; ++c) s[4 * i + c] = __fadd_rn(pR[4 * i + c], f4(f, c));
        }
        thT = row_theta<NL, KP>(s, top_b, half, lane, jT);
        if (st) {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float4 f = lds4(sg[8 + i][x]);
#pragma unroll
                for (int c = 0; c < 4; ++c) s[4 * i + c] = __fadd_rn(s[4 * i + c], f4(f, c));
            }
            thST = row_theta<NL, KP>(s, top_b, half, lane, jST);
        }
    }
    const float k2 = a.k2;
    float lT = 0.f, WT = 0.f, lST = 0.f, WST = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const float4 fT = lds4(sg[i][x]), fq = lds4(sg[4 + i][x]);
        const float4 fS = st ? lds4(sg[8 + i][x]) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
        for (int c = 0; c < 4; ++c) {
            const int j = 4 * i + c;
            const float q = f4(fq, c);
            const float sT = __fadd_rn(pR[j], f4(fT, c));
            // with d = s - theta, u = sigmoid(|d| / tau), v = 1 - u: 1 - m = v if
            // d >= 0 else u, and w = q m (1 - m) = q u v
            const float d = sT - thT;
            const float E = ex2_approx(-fabsf(d) * k2);
            const float u = rcp_approx(1.f + E);
            const float v = E * u;
            const float om = d >= 0.f ? v : u;
            lT = fmaf(q, om, lT);
            const float w = q * (u * v);
            WT += w;
            float omS = 0.f, wS = 0.f;
            if (st) {
                const float d2 = __fadd_rn(sT, f4(fS, c)) - thST;
                const float E2 = ex2_approx(-fabsf(d2) * k2);
                const float u2 = rcp_approx(1.f + E2);
                const float v2 = E2 * u2;
                omS = d2 >= 0.f ? v2 : u2;
                lST = fmaf(q, omS, lST);
                wS = q * (u2 * v2);
                WST += wS;
            }
            const float gs = -fmaf(a.gT, w, a.gST * wS);
            dT[j] = gs;
            dR[j] = carry[j] + gs;
            dS[j] = -a.gST * wS;
            carry[j] = fmaf(a.cT, om, a.cST * omS);
        }
    }
    lT = pair_sum<NL>(lT);
    WT = pair_sum<NL>(WT);
    lST = pair_sum<NL>(lST);
    WST = pair_sum<NL>(WST);
    // through theta_B = s_{e*}: dl/ds_{e*} gains W / tau
    const float cw = a.gT * WT, cws = a.gST * WST;
#pragma unroll
    for (int j = 0; j < kRowE; ++j) {
        const float add = (j == jT ? cw : 0.f) + (j == jST ? cws : 0.f);
        dT[j] += add;
        dR[j] += add;
        dS[j] += j == jST ? cws : 0.f;
    }
    return make_float2(lT, lST);
}

template <int NL, int KP, bool ST>
__global__ void __launch_bounds__(32 * kRowWarps, 3) cache_loss_rows_kernel(const LossArgs a) {
    constexpr int CPW = 32 / NL;                         // tasks per warp
    const int lane = threadIdx.x & 31;
    const int half = NL == 2 ? (lane & 1) : 0;
    const int warp = blockIdx.x * kRowWarps + (threadIdx.x >> 5);
    const int BL = a.B * a.L;
    const int wpc = (BL + CPW - 1) / CPW;                // warps per token chunk
    if (warp >= wpc * a.nchunks) return;                 // whole warps
    const int c = warp / wpc;
    const int jl = (warp % wpc) * CPW + lane / NL;       // b * L + l
    const bool active = jl < BL;                         // idle pairs run on zeros
    const int T = a.T, L = a.L, N = a.N;
    const int b = active ? jl / L : 0, l = active ? jl % L : 0;
    const int t0 = c * a.chunk;
    const int t1 = min(T, t0 + a.chunk);
    constexpr bool st = ST;
    const bool wr = active && a.grad != nullptr;
    const size_t row3 = (size_t)3 * N;
    const size_t tok = (size_t)L * row3;
    const size_t base = ((size_t)b * T * L + l) * row3 + (size_t)half * kRowE;
    const size_t s_off = l > 0 ? tok + (size_t)2 * N - row3 : (size_t)(L - 1 - l) * row3 + 2 * N;
    const float* pp = a.probs + base + (size_t)t0 * tok;
    float* gp = a.grad ? a.grad + base + (size_t)t0 * tok : nullptr;
    float* lossp = (a.loss && active && half == 0)
                       ? a.loss + (((size_t)b * T + t0) * L + l) * 2 : nullptr;

    // The rows of step t are copied into shared memory one step ahead
    // (cp.async, two stages); each warp's accesses to a stage are contiguous.
    __shared__ RowStage stg[2];
    const int x = threadIdx.x;
    auto prefetch = [&](int k, const float* u, int t) {       // u: unit (b, t, l)
        const bool nx = active && t + 1 < T;
#pragma unroll
        for (int i = 0; i < 4; ++i) cp_async16(&stg[k][i][x], u + N + 4 * i, active);
#pragma unroll
        for (int i = 0; i < 4; ++i) cp_async16(&stg[k][4 + i][x], nx ? u + tok + 4 * i : u, nx);
        if (st) {
#pragma unroll
            for (int i = 0; i < 4; ++i)
                cp_async16(&stg[k][8 + i][x], nx ? u + s_off + 4 * i : u, nx);
        }
        cp_async_commit();
    };
    auto take_q = [&](float (&v)[kRowE], int k) {       // p^R_{t+1} of stage k
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float4 f = lds4(stg[k][4 + i][x]);
            v[4 * i] = f.x;
            v[4 * i + 1] = f.y;
            v[4 * i + 2] = f.z;
            v[4 * i + 3] = f.w;
        }
    };

    float pR[kRowE], carry[kRowE];
    float dR[kRowE], dT[kRowE], dS[kRowE];
#pragma unroll
    for (int j = 0; j < kRowE; ++j) carry[j] = 0.f;
    double sumT = 0.0, sumST = 0.0;
    prefetch(0, pp, t0);

    if (t0 > 0) {
        // halo: the terms of step t0 - 1 give the target part of p^R_{t0}
        prefetch(1, pp - tok, t0 - 1);
        asm volatile("cp.async.wait_group 0;" ::: "memory");
        load16(pR, pp - tok, active);
        rows_step<NL, KP>(pR, stg[1], x, st, a.top_b, a, half, lane, carry, dR, dT, dS);
        take_q(pR, 1);
    } else {
        load16(pR, pp, active);
        if (lossp) lossp[1] = 0.f;                       // no l^ST at t = 0
        if (st && wr && l > 0) {                         // p^S of rho(0, l) receives nothing
            float z[kRowE];
#pragma unroll
            for (int j = 0; j < kRowE; ++j) z[j] = 0.f;
            store16(gp + 2 * N - row3, z);
        }
    }

#pragma unroll 1
    for (int t = t0; t < t1; ++t, pp += tok) {
        const int k = (t - t0) & 1;
        if (t + 1 < t1)
            prefetch(k ^ 1, pp + tok, t + 1);
        else
            cp_async_commit();                           // an empty group keeps the count
        cp_async_wait1();                                // this step's copies have landed
        const bool next = t + 1 < T;
        if (next) {
            const float2 y =
                rows_step<NL, KP>(pR, stg[k], x, st, a.top_b, a, half, lane, carry, dR, dT, dS);
            sumT += (double)y.x;
            sumST += (double)y.y;
            if (lossp) {
                lossp[0] = y.x;
                lossp[(size_t)L * 2 + 1] = st ? y.y : 0.f;
            }
        } else {
            // last token: no l^T here, no l^ST after it
            if (lossp) lossp[0] = 0.f;
#pragma unroll
            for (int j = 0; j < kRowE; ++j) {
                dR[j] = carry[j];
                dT[j] = dS[j] = 0.f;
            }
            if (st && wr && l == 0) {                    // p^S of rho(T, 0) receives nothing
                float z[kRowE];
#pragma unroll
                for (int j = 0; j < kRowE; ++j) z[j] = 0.f;
                store16(gp + s_off, z);
            }
        }
        if (a.grad) {
            // softmax backward of each head row: dz = p (dp - <p, dp>)
            const bool ws = st && next;
            float xR = 0.f, xT = 0.f, xS = 0.f;
#pragma unroll
            for (int i = 0; i < 4; ++i) {
                const float4 fT = lds4(stg[k][i][x]);
                const float4 fS = ws ? lds4(stg[k][8 + i][x]) : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int c = 0; c < 4; ++c) {
                    const int j = 4 * i + c;
                    xR = fmaf(pR[j], dR[j], xR);
                    xT = fmaf(f4(fT, c), dT[j], xT);
                    xS = fmaf(f4(fS, c), dS[j], xS);
                }
            }
            xR = pair_sum<NL>(xR);
            xT = pair_sum<NL>(xT);
            xS = pair_sum<NL>(xS);
            if (wr) {
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const int j = 4 * i;
                    __stcs(reinterpret_cast<float4*>(gp) + i,
                           make_float4(pR[j] * (dR[j] - xR), pR[j + 1] * (dR[j + 1] - xR),
                                       pR[j + 2] * (dR[j + 2] - xR), pR[j + 3] * (dR[j + 3] - xR)));
                    const float4 fT = lds4(stg[k][i][x]);
                    __stcs(reinterpret_cast<float4*>(gp + N) + i,
                           make_float4(fT.x * (dT[j] - xT), fT.y * (dT[j + 1] - xT),
                                       fT.z * (dT[j + 2] - xT), fT.w * (dT[j + 3] - xT)));
                    if (ws) {
                        const float4 fS = lds4(stg[k][8 + i][x]);
                        __stcs(reinterpret_cast<float4*>(gp + s_off) + i,
                               make_float4(fS.x * (dS[j] - xS), fS.y * (dS[j + 1] - xS),
                                           fS.z * (dS[j + 2] - xS), fS.w * (dS[j + 3] - xS)));
                    }
                }
            }
            gp += tok;
        }
        if (lossp) lossp += (size_t)L * 2;
        if (next) take_q(pR, k);
    }
    if (a.partial && active && half == 0) {
        const size_t task = ((size_t)b * a.nchunks + c) * L + l;
        a.partial[task * 2 + 0] = sumT;
        a.partial[task * 2 + 1] = sumST;
    }
}

// Token chunks of the short-row kernel: as many as give every resident warp
// one (a single wave, each warp running one chunk of its 32 / NL chains),
// chunks of at least 32 tokens so the halo step costs <= 1/32.
template <int NL, int KP, bool ST>
int launch_loss_rows(LossArgs& a, cudaStream_t stream) {
    constexpr int CPW = 32 / NL;
    static std::atomic<int> blocks_per_sm{0};
    if (blocks_per_sm.load() == 0) {
        int n = 0;
        if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, cache_loss_rows_kernel<NL, KP, ST>,
                                                          32 * kRowWarps, 0) != cudaSuccess)
            return CRC_ECUDA;
        blocks_per_sm.store(n > 0 ? n : 1);
    }
    const long long groups = (a.B * (long long)a.L + CPW - 1) / CPW;
    const long long resident = (long long)sm_count() * blocks_per_sm.load() * kRowWarps;
    long long n = resident / groups;
    const long long cap = (a.T + 31) / 32;
    if (n > cap) n = cap;
    if (n < 1) n = 1;
    a.chunk = (int)((a.T + n - 1) / n);
    a.nchunks = (a.T + a.chunk - 1) / a.chunk;
    const long long warps = groups * a.nchunks;
    const int grid = (int)((warps + kRowWarps - 1) / kRowWarps);
    {
        ProfScope prof(CRC_KERNEL_LOSS, stream);
        cache_loss_rows_kernel<NL, KP, ST><<<grid, 32 * kRowWarps, 0, stream>>>(a);
    }
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

template <int NL, bool ST>
int launch_loss_rows_st(LossArgs& a, cudaStream_t stream) {
    if (a.top_b <= 2) return launch_loss_rows<NL, 2, ST>(a, stream);
    if (a.top_b <= 4) return launch_loss_rows<NL, 4, ST>(a, stream);
    if (a.top_b <= 8) return launch_loss_rows<NL, 8, ST>(a, stream);
    return launch_loss_rows<NL, 16, ST>(a, stream);
}

template <int NL>
int launch_loss_rows_kp(LossArgs& a, cudaStream_t stream) {
    return a.heads == 3 ? launch_loss_rows_st<NL, true>(a, stream)
                        : launch_loss_rows_st<NL, false>(a, stream);
}

// Means L_T, L_ST: fixed-order sums of the per-task sums (deterministic).
constexpr int kMeanThreads = 256;

__global__ void __launch_bounds__(kMeanThreads)
    loss_means_kernel(const double* partial, int tasks, double inv_nT, double inv_nST,
                      double* means) {
    __shared__ double sh[2][kMeanThreads];
    double aT = 0.0, aST = 0.0;
    for (int i = threadIdx.x; i < tasks; i += kMeanThreads) {
        aT += partial[(size_t)i * 2 + 0];
        aST += partial[(size_t)i * 2 + 1];
    }
    sh[0][threadIdx.x] = aT;
    sh[1][threadIdx.x] = aST;
    __syncthreads();
    for (int w = kMeanThreads / 2; w > 0; w >>= 1) {
        if ((int)threadIdx.x < w) {
            sh[0][threadIdx.x] += sh[0][threadIdx.x + w];
            sh[1][threadIdx.x] += sh[1][threadIdx.x + w];
        }
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        means[0] = sh[0][0] * inv_nT;
        means[1] = sh[1][0] * inv_nST;
    }
}

template <int V, bool ALL_VALID>
int launch_loss_t(const LossArgs& a, cudaStream_t stream) {
    const int tasks = a.B * a.L * a.nchunks;
    const int grid = (tasks + kLossWarps - 1) / kLossWarps;
    {
        ProfScope prof(CRC_KERNEL_LOSS, stream);
        if (a.heads == 3)
            cache_loss_kernel<V, ALL_VALID, true><<<grid, 32 * kLossWarps, 0, stream>>>(a);
        else
            cache_loss_kernel<V, ALL_VALID, false><<<grid, 32 * kLossWarps, 0, stream>>>(a);
    }
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

}  // namespace

long long loss_task_slots(int B, int L, int T, int N) {
    const long long bl = (long long)B * L;
    if (T <= 0) return 0;
    if (N <= 32) return bl * ((T + 31) / 32);
    return bl * loss_plan(B, L, T).nchunks;
}

LossPlan loss_plan(int B, int L, int T) {
    // About 49152 warp tasks (ten waves of resident warps on a 152-SM GPU,
    // so the last one idles little), chunks of at least 32 tokens so the halo
    // step costs <= 1/32.
    LossPlan pl{1, T > 0 ? T : 1};
    if (T <= 0) return pl;
    const long long bl = (long long)B * L;
    long long n = (49152 + bl - 1) / bl;
    const long long cap = (T + 31) / 32;
    if (n > cap) n = cap;
    if (n < 1) n = 1;
    pl.chunk = (int)((T + n - 1) / n);
    pl.nchunks = (T + pl.chunk - 1) / pl.chunk;
    return pl;
}

int launch_cache_loss(const crc_problem& p, const float* probs, int T, int heads, int top_b,
                      double tau, double w_T, double w_ST, float* loss, double* means,
                      float* grad, void* workspace, cudaStream_t stream) {
    const LossPlan pl = loss_plan(p.B, p.L, T);
    const double n_valid = (double)p.B * (double)(T - 1) * (double)p.L;   // |Omega_T| = |Omega_ST|
    LossArgs a;
    a.probs = probs;
    a.loss = loss;
    a.grad = grad;
    a.partial = means ? static_cast<double*>(workspace) : nullptr;
    a.B = p.B;
    a.T = T;
    a.L = p.L;
    a.N = p.N;
    a.heads = heads;
    a.top_b = top_b;
    a.chunk = pl.chunk;
    a.nchunks = pl.nchunks;
    a.k2 = (float)(1.4426950408889634 / tau);
    const double cT = n_valid > 0 ? w_T / n_valid : 0.0;
    const double cST = n_valid > 0 && heads == 3 ? w_ST / n_valid : 0.0;
    a.cT = (float)cT;
    a.cST = (float)cST;
    a.gT = (float)(cT / tau);
    a.gST = (float)(cST / tau);
    int rc;
    if ((p.N == 16 || p.N == 32) && top_b <= 16) {
        // short rows: 16 elements per lane, one or two lanes per row
        rc = p.N == 16 ? launch_loss_rows_kp<1>(a, stream) : launch_loss_rows_kp<2>(a, stream);
    } else {
#define CRC_LOSS_V(VV)                                                               \
    rc = p.N == 32 * VV ? launch_loss_t<VV, true>(a, stream)                         \
                        : launch_loss_t<VV, false>(a, stream);
    if (p.N <= 32) {
        CRC_LOSS_V(1)
    } else if (p.N <= 64) {
        CRC_LOSS_V(2)
    } else if (p.N <= 128) {
        CRC_LOSS_V(4)
    } else {
        CRC_LOSS_V(8)
    }
#undef CRC_LOSS_V
    }
    if (rc != CRC_OK || !means) return rc;
    const double inv_n = n_valid > 0 ? 1.0 / n_valid : 0.0;
    {
        ProfScope prof(CRC_KERNEL_LOSS_MEANS, stream);
        loss_means_kernel<<<1, kMeanThreads, 0, stream>>>(
            static_cast<const double*>(workspace), p.B * p.L * a.nchunks, inv_n,
            heads == 3 ? inv_n : 0.0, means);
    }
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

}  // namespace crc
