// Fused route-and-cache: workspace size and dispatch on N.
#include "fused_launch.cuh"

namespace crc {

size_t fused_workspace_bytes(const crc_problem& p) { return fused_plan(p, 0).total; }

int launch_fused(const crc_problem& p, const uint16_t* hidden, const uint16_t* w_cat, int T,
                 void* state, void* workspace, size_t workspace_bytes, const crc_trace* trace,
                 cudaStream_t stream) {
    if (p.K > 8 || workspace_bytes < fused_workspace_bytes(p)) return CRC_EUNSUPPORTED;
    switch (p.N) {
        case 16: return launch_fused_n16(p, hidden, w_cat, T, state, workspace, trace, stream);
        case 32: return launch_fused_n32(p, hidden, w_cat, T, state, workspace, trace, stream);
        case 64: return launch_fused_n64(p, hidden, w_cat, T, state, workspace, trace, stream);
        case 128: return launch_fused_n128(p, hidden, w_cat, T, state, workspace, trace, stream);
        default: return CRC_EUNSUPPORTED;
    }
}

}  // namespace crc
