// Launch of the comparison-policy cache scan (policy_scan.cuh) for one
// policy; each policy's instantiations sit in a translation unit of their own
// (policy_lru.cu, policy_lfu.cu, policy_lrfu.cu, policy_spatio.cu) so that
// they compile in parallel, and policy.cu dispatches on the policy.
#pragma once

#include "crc_internal.h"
#include "policy_scan.cuh"

namespace crc {

template <int V, bool ALL_VALID, int KP, int POL>
int launch_policy_t(const crc_problem& p, const float* scores, int T, void* state,
                    const crc_trace* trace, int trace_T, int trace_t0, int lambda2,
                    cudaStream_t stream) {
    PolicyArgs a;
    a.s.scores = scores;
    a.s.state = static_cast<uint8_t*>(state);
    a.s.B = p.B;
    a.s.T = T;
    a.s.L = p.L;
    a.s.N = p.N;
    a.s.K = p.K;
    a.s.C = p.C;
    a.s.R = p.R;
    a.s.trace_T = trace_T;
    a.s.trace_t0 = trace_t0;
    a.s.trace_topk = trace ? trace->topk_dev : nullptr;
    a.s.trace_miss = trace ? trace->misses_dev : nullptr;
    a.s.trace_pro = trace ? trace->proactive_dev : nullptr;
    a.s.trace_mid = nullptr;                     // cache traces: the method's scan only
    a.s.trace_after = nullptr;
    a.s.trace_sel = nullptr;
    a.policy = POL;
    a.lambda2 = lambda2;
    const int chains = p.B * p.L;
    const int warps_per_block = kScanWarps;
    const int grid = (chains + warps_per_block - 1) / warps_per_block;
    {
        ProfScope prof(CRC_KERNEL_SCAN, stream);
        cache_scan_policy_kernel<V, ALL_VALID, KP, POL>
            <<<grid, 32 * warps_per_block, 0, stream>>>(a);
    }
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

template <int POL>
int launch_policy_pol(const crc_problem& p, const float* scores, int T, void* state,
                      const crc_trace* trace, int trace_T, int trace_t0, int lambda2,
                      cudaStream_t stream) {
#define CRC_POLICY_KP(VV, KPV)                                                              \
    return p.N == 32 * VV                                                                   \
               ? launch_policy_t<VV, true, KPV, POL>(p, scores, T, state, trace, trace_T,   \
                                                     trace_t0, lambda2, stream)             \
               : launch_policy_t<VV, false, KPV, POL>(p, scores, T, state, trace, trace_T,  \
                                                      trace_t0, lambda2, stream);
#define CRC_POLICY_V(VV)                    \
    {                                       \
        if (p.K <= 2) CRC_POLICY_KP(VV, 2)  \
        if (p.K <= 4) CRC_POLICY_KP(VV, 4)  \
        if (p.K <= 8) CRC_POLICY_KP(VV, 8)  \
        if (p.K <= 16) CRC_POLICY_KP(VV, 16) \
        CRC_POLICY_KP(VV, 32)               \
    }
    if (p.N <= 32) CRC_POLICY_V(1)
    if (p.N <= 64) CRC_POLICY_V(2)
    if (p.N <= 128) CRC_POLICY_V(4)
    CRC_POLICY_V(8)
#undef CRC_POLICY_V
#undef CRC_POLICY_KP
}

}  // namespace crc
