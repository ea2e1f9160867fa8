// The method's cache-scan kernels with trace writes (scan_launch.cuh).
#include "scan_launch.cuh"

namespace crc {
template int launch_scan_mode<true>(const crc_problem&, const float*, int, void*,
                                    const crc_trace*, int, int, cudaStream_t);
}  // namespace crc
