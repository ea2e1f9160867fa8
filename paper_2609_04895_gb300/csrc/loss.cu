// Soft Top-B cache-coverage losses and their gradient (Sec. 3.1-3.4), from the
// router probabilities, one warp per (stream, layer, token chunk).
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

#include "crc_internal.h"

namespace crc {
namespace {

constexpr unsigned kFull = 0xffffffffu;
constexpr int kLossWarps = 8;

struct LossArgs {
    const float* probs;   // [B][T][L][3][N]
    float* loss;          // [B][T][L][2] (l^T, l^ST) or null
    float* grad;          // [B][T][L][3][N] or null
    double* partial;      // [tasks][2] per-task sums of l^T and l^ST, or null
    int B, T, L, N, heads, top_b, chunk, nchunks;
    float inv_tau, cT, cST;
};

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFull, v, o);
    return v;
}

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
    const int rank = top_b - (int)__reduce_add_sync(kFull, gt);   // 1-based among the equal keys
    const uint32_t neq = __reduce_add_sync(kFull, eq);
    int before = 0;
    if (neq > 1u) {                                 // ties at theta: exclusive scan of eq
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

// One coverage term l(s, q): returns the loss, writes g = dl/ds and gq = dl/dq.
template <int V>
__device__ __forceinline__ float coverage(const float (&s)[V], const float (&q)[V], bool valid,
                                          int top_b, float inv_tau, int lane, float (&g)[V],
                                          float (&gq)[V]) {
    uint32_t k[V];
#pragma unroll
    for (int j = 0; j < V; ++j) k[j] = valid ? __float_as_uint(s[j]) : 0u;
    const uint32_t th = theta_key<V>(k, valid, top_b);
    const int js = theta_slot<V>(k, valid, th, top_b, lane);
    const float theta = __uint_as_float(th);
    float loss = 0.f, sdm = 0.f;
#pragma unroll
    for (int j = 0; j < V; ++j) {
        const float x = (s[j] - theta) * inv_tau;
        const float E = __expf(-fabsf(x));             // in (0, 1]
        const float up = __fdividef(1.f, 1.f + E);      // sigmoid(|x|)
        const float dn = E * up;                        // sigmoid(-|x|)
        const float om = x >= 0.f ? dn : up;            // 1 - m_e
        loss = fmaf(q[j], om, loss);
        const float dm = q[j] * (up * dn) * inv_tau;    // q_e dm_e/ds_e
        g[j] = -dm;
        gq[j] = om;
        sdm += dm;
    }
    loss = warp_sum(loss);
    sdm = warp_sum(sdm);
#pragma unroll
    for (int j = 0; j < V; ++j)
        if (j == js) g[j] += sdm;                       // through theta_B = s_{e*}
    return loss;
}

// Softmax backward of one head row and its store: dz = p (dp - <p, dp>).
template <int V>
__device__ __forceinline__ void store_dz(float* row, const float (&p)[V], const float (&d)[V],
                                         int lane, bool valid) {
    float dot = 0.f;
#pragma unroll
    for (int j = 0; j < V; ++j) dot = fmaf(p[j], d[j], dot);
    dot = warp_sum(dot);
    float o[V];
#pragma unroll
    for (int j = 0; j < V; ++j) o[j] = p[j] * (d[j] - dot);
    store_row<V>(row, o, lane, valid);
}

template <int V>
__device__ __forceinline__ void store_zero(float* row, int lane, bool valid) {
    float z[V];
#pragma unroll
    for (int j = 0; j < V; ++j) z[j] = 0.f;
    store_row<V>(row, z, lane, valid);
}

template <int V, bool ALL_VALID>
__global__ void __launch_bounds__(32 * kLossWarps) cache_loss_kernel(const LossArgs a) {
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
    const bool st = a.heads == 3;
    const bool want_grad = a.grad != nullptr;
    const size_t row3 = (size_t)3 * N;
    const size_t u_b = (size_t)b * T;
    auto unit = [&](int t, int ll) { return (u_b + t) * L + ll; };
    auto prow = [&](int t, int ll, int h) { return a.probs + unit(t, ll) * row3 + (size_t)h * N; };
    auto grow = [&](int t, int ll, int h) { return a.grad + unit(t, ll) * row3 + (size_t)h * N; };
    // rho(t + 1, l): (t, L - 1) for l = 0, (t + 1, l - 1) otherwise
    auto srow = [&](int t) { return l > 0 ? prow(t + 1, l - 1, 2) : prow(t, L - 1, 2); };
    auto sgrow = [&](int t) { return l > 0 ? grow(t + 1, l - 1, 2) : grow(t, L - 1, 2); };

    float pR[V], pT[V], q[V], pS[V], carry[V];
    float gT[V], gqT[V], gST[V], gqST[V];
#pragma unroll
    for (int j = 0; j < V; ++j) {
        carry[j] = 0.f;
        gST[j] = gqST[j] = pS[j] = 0.f;
    }
    double sumT = 0.0, sumST = 0.0;

    if (t0 > 0) {
        // halo: the two terms of step t0 - 1 give the target part of p^R_{t0}
        load_row<V>(pR, prow(t0 - 1, l, 0), lane, valid);
        load_row<V>(pT, prow(t0 - 1, l, 1), lane, valid);
        load_row<V>(q, prow(t0, l, 0), lane, valid);
        if (st) load_row<V>(pS, srow(t0 - 1), lane, valid);
        float s[V];
#pragma unroll
        for (int j = 0; j < V; ++j) s[j] = __fadd_rn(pR[j], pT[j]);
        coverage<V>(s, q, valid, a.top_b, a.inv_tau, lane, gT, gqT);
        if (st) {
#pragma unroll
            for (int j = 0; j < V; ++j) s[j] = __fadd_rn(s[j], pS[j]);
            coverage<V>(s, q, valid, a.top_b, a.inv_tau, lane, gST, gqST);
        }
#pragma unroll
        for (int j = 0; j < V; ++j) {
            carry[j] = a.cT * gqT[j] + a.cST * gqST[j];
            pR[j] = q[j];
        }
    } else {
        load_row<V>(pR, prow(0, l, 0), lane, valid);
        if (a.loss && lane == 0) a.loss[unit(0, l) * 2 + 1] = 0.f;     // no l^ST at t = 0
        if (st && want_grad && l > 0) store_zero<V>(grow(0, l - 1, 2), lane, valid);
    }

#pragma unroll 1
    for (int t = t0; t < t1; ++t) {
        load_row<V>(pT, prow(t, l, 1), lane, valid);
        float dR[V], dT[V];
        if (t + 1 < T) {
            load_row<V>(q, prow(t + 1, l, 0), lane, valid);
            if (st) load_row<V>(pS, srow(t), lane, valid);
            float s[V];
#pragma unroll
            for (int j = 0; j < V; ++j) s[j] = __fadd_rn(pR[j], pT[j]);
            const float lT = coverage<V>(s, q, valid, a.top_b, a.inv_tau, lane, gT, gqT);
            float lST = 0.f;
            if (st) {
#pragma unroll
                for (int j = 0; j < V; ++j) s[j] = __fadd_rn(s[j], pS[j]);
                lST = coverage<V>(s, q, valid, a.top_b, a.inv_tau, lane, gST, gqST);
            }
            sumT += (double)lT;
            sumST += (double)lST;
            if (a.loss && lane == 0) {
                a.loss[unit(t, l) * 2 + 0] = lT;
                a.loss[unit(t + 1, l) * 2 + 1] = st ? lST : 0.f;
            }
#pragma unroll
            for (int j = 0; j < V; ++j) {
                const float gs = a.cT * gT[j] + a.cST * gST[j];
                dT[j] = gs;
                dR[j] = carry[j] + gs;
                carry[j] = a.cT * gqT[j] + a.cST * gqST[j];
            }
            if (st && want_grad) {
                float dS[V];
#pragma unroll
                for (int j = 0; j < V; ++j) dS[j] = a.cST * gST[j];
                store_dz<V>(sgrow(t), pS, dS, lane, valid);
            }
        } else {
            // last token: no l^T here, no l^ST after it
            if (a.loss && lane == 0) a.loss[unit(t, l) * 2 + 0] = 0.f;
#pragma unroll
            for (int j = 0; j < V; ++j) {
                dR[j] = carry[j];
                dT[j] = 0.f;
            }
            if (st && want_grad && l == 0) store_zero<V>(grow(t, L - 1, 2), lane, valid);
        }
        if (want_grad) {
            store_dz<V>(grow(t, l, 0), pR, dR, lane, valid);
            store_dz<V>(grow(t, l, 1), pT, dT, lane, valid);
        }
#pragma unroll
        for (int j = 0; j < V; ++j) pR[j] = q[j];
    }
    if (a.partial && lane == 0) {
        a.partial[(size_t)task * 2 + 0] = sumT;
        a.partial[(size_t)task * 2 + 1] = sumST;
    }
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
        cache_loss_kernel<V, ALL_VALID><<<grid, 32 * kLossWarps, 0, stream>>>(a);
    }
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

}  // namespace

LossPlan loss_plan(int B, int L, int T) {
    // About 8192 warp tasks (several waves of resident warps on any current
    // GPU), chunks of at least 16 tokens so the halo step costs <= 1/16.
    LossPlan pl{1, T > 0 ? T : 1};
    if (T <= 0) return pl;
    const long long bl = (long long)B * L;
    long long n = (8192 + bl - 1) / bl;
    const long long cap = (T + 15) / 16;
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
    a.inv_tau = (float)(1.0 / tau);
    a.cT = n_valid > 0 ? (float)(w_T / n_valid) : 0.f;
    a.cST = n_valid > 0 && heads == 3 ? (float)(w_ST / n_valid) : 0.f;
    int rc;
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
    if (rc != CRC_OK || !means) return rc;
    const double inv_n = n_valid > 0 ? 1.0 / n_valid : 0.0;
    {
        ProfScope prof(CRC_KERNEL_LOSS_MEANS, stream);
        loss_means_kernel<<<1, kMeanThreads, 0, stream>>>(
            static_cast<const double*>(workspace), p.B * p.L * pl.nchunks, inv_n,
            heads == 3 ? inv_n : 0.0, means);
    }
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

}  // namespace crc
