// The comparison-policy scan's instantiations for CRC_POLICY_SPATIO_LRU.
#include "policy_launch.cuh"

namespace crc {
template int launch_policy_pol<CRC_POLICY_SPATIO_LRU>(const crc_problem&, const float*, int, void*,
                                       const crc_trace*, int, int, int, cudaStream_t);
}  // namespace crc
