// Launch of the method's cache-scan kernel for one trace mode; the untraced
// kernels are instantiated in scan.cu, the traced ones in scan_traced.cu, so
// that the two compile in parallel.
#pragma once

#include "cache_scan.cuh"
#include "crc_internal.h"

namespace crc {

template <int V, bool ALL_VALID, int KP, bool TRACED>
int launch_scan_t(const crc_problem& p, const float* scores, int T, void* state,
                  const crc_trace* trace, int trace_T, int trace_t0, cudaStream_t stream) {
    ScanArgs a;
    a.scores = scores;
    a.state = static_cast<uint8_t*>(state);
    a.B = p.B;
    a.T = T;
    a.L = p.L;
    a.N = p.N;
    a.K = p.K;
    a.C = p.C;
    a.R = p.R;
    a.trace_T = trace_T;
    a.trace_t0 = trace_t0;
    a.trace_topk = trace ? trace->topk_dev : nullptr;
    a.trace_miss = trace ? trace->misses_dev : nullptr;
    a.trace_pro = trace ? trace->proactive_dev : nullptr;
    a.trace_mid = trace ? trace->cache_mid_dev : nullptr;
    a.trace_after = trace ? trace->cache_after_dev : nullptr;
    a.trace_sel = trace ? trace->topk_set_dev : nullptr;
    const int chains = p.B * p.L;
    const int warps_per_block = kScanWarps;
    const int grid = (chains + warps_per_block - 1) / warps_per_block;
    {
        ProfScope prof(CRC_KERNEL_SCAN, stream);
        cache_scan_kernel<V, ALL_VALID, KP, TRACED><<<grid, 32 * warps_per_block, 0, stream>>>(a);
    }
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

template <bool TRACED>
int launch_scan_mode(const crc_problem& p, const float* scores, int T, void* state,
                     const crc_trace* trace, int trace_T, int trace_t0, cudaStream_t stream) {
#define CRC_SCAN_KP(VV, KPV)                                                                  \
    return (p.N == 32 * VV)                                                                  \
               ? launch_scan_t<VV, true, KPV, TRACED>(p, scores, T, state, trace, trace_T,    \
                                                      trace_t0, stream)                       \
               : launch_scan_t<VV, false, KPV, TRACED>(p, scores, T, state, trace, trace_T,   \
                                                       trace_t0, stream);
#define CRC_SCAN(VV)                      \
    {                                     \
        if (p.K <= 2) CRC_SCAN_KP(VV, 2)  \
        if (p.K <= 4) CRC_SCAN_KP(VV, 4)  \
        if (p.K <= 8) CRC_SCAN_KP(VV, 8)  \
        if (p.K <= 16) CRC_SCAN_KP(VV, 16) \
        CRC_SCAN_KP(VV, 32)               \
    }
    if (p.N <= 32) CRC_SCAN(1)
    if (p.N <= 64) CRC_SCAN(2)
    if (p.N <= 128) CRC_SCAN(4)
    CRC_SCAN(8)
#undef CRC_SCAN_KP
#undef CRC_SCAN
}

}  // namespace crc
