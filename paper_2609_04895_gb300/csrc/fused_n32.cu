// Fused route-and-cache instantiations for N = 32 experts per layer.
#include "fused_launch.cuh"

namespace crc {

int launch_fused_n32(const crc_problem& p, const uint16_t* hidden, const uint16_t* w_cat, int T,
                     void* state, void* workspace, const crc_trace* trace,
                     cudaStream_t stream) {
    return launch_fused_for_n<32, 1, true>(p, hidden, w_cat, T, state, workspace, trace, stream);
}

}  // namespace crc
