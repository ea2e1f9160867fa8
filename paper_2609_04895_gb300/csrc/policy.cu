// Dispatch of the comparison-policy cache scan (policy_scan.cuh) on the
// policy; each policy's kernels are instantiated in policy_<name>.cu.
#include "crc_internal.h"

namespace crc {

template <int POL>
int launch_policy_pol(const crc_problem& p, const float* scores, int T, void* state,
                      const crc_trace* trace, int trace_T, int trace_t0, int lambda2,
                      cudaStream_t stream);

int launch_policy_scan(const crc_problem& p, const float* scores, int T, void* state,
                       const crc_trace* trace, int trace_T, int trace_t0, int policy,
                       int lambda2, cudaStream_t stream) {
    if (T <= 0) return CRC_OK;
    switch (policy) {
    case CRC_POLICY_LRU:
        return launch_policy_pol<CRC_POLICY_LRU>(p, scores, T, state, trace, trace_T, trace_t0,
                                                 lambda2, stream);
    case CRC_POLICY_LFU:
        return launch_policy_pol<CRC_POLICY_LFU>(p, scores, T, state, trace, trace_T, trace_t0,
                                                 lambda2, stream);
    case CRC_POLICY_LRFU:
        return launch_policy_pol<CRC_POLICY_LRFU>(p, scores, T, state, trace, trace_T, trace_t0,
                                                  lambda2, stream);
    case CRC_POLICY_SPATIO_LRU:
        return launch_policy_pol<CRC_POLICY_SPATIO_LRU>(p, scores, T, state, trace, trace_T,
                                                        trace_t0, lambda2, stream);
    default:
        return CRC_EINVAL;
    }
}

}  // namespace crc
