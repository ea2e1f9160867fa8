// The comparison-policy scan's instantiations for CRC_POLICY_LFU.
#include "policy_launch.cuh"

namespace crc {
template int launch_policy_pol<CRC_POLICY_LFU>(const crc_problem&, const float*, int, void*,
                                       const crc_trace*, int, int, int, cudaStream_t);
}  // namespace crc
