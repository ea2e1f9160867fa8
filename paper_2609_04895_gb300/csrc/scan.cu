// Host launcher of the cache-scan kernel (the untraced instantiations; the
// traced ones are in scan_traced.cu) and the state initialiser.
#include "scan_launch.cuh"

namespace crc {
namespace {

// Writes the header of a state whose bytes were zeroed just before.
__global__ void state_init_kernel(uint8_t* state, crc_problem p) {
    StateHeader* h = reinterpret_cast<StateHeader*>(state);
    h->magic = kStateMagic;
    h->L = p.L;
    h->N = p.N;
    h->K = p.K;
    h->C = p.C;
    h->R = p.R;
    h->B = p.B;
    h->expert_bytes = p.expert_bytes;
}

}  // namespace

int launch_state_init(const crc_problem& p, void* state, size_t bytes, cudaStream_t stream) {
    if (cudaMemsetAsync(state, 0, bytes, stream) != cudaSuccess) return CRC_ECUDA;
    {
        ProfScope prof(CRC_KERNEL_STATE, stream);
        state_init_kernel<<<1, 1, 0, stream>>>(static_cast<uint8_t*>(state), p);
    }
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}

template int launch_scan_mode<false>(const crc_problem&, const float*, int, void*,
                                     const crc_trace*, int, int, cudaStream_t);
extern template int launch_scan_mode<true>(const crc_problem&, const float*, int, void*,
                                           const crc_trace*, int, int, cudaStream_t);

int launch_scan(const crc_problem& p, const float* scores, int T, void* state,
                const crc_trace* trace, int trace_T, int trace_t0, cudaStream_t stream) {
    if (T <= 0) return CRC_OK;
    const bool traced = trace && (trace->topk_dev || trace->misses_dev || trace->proactive_dev ||
                                  trace->cache_mid_dev || trace->cache_after_dev ||
                                  trace->topk_set_dev);
    return traced ? launch_scan_mode<true>(p, scores, T, state, trace, trace_T, trace_t0, stream)
                  : launch_scan_mode<false>(p, scores, T, state, trace, trace_T, trace_t0, stream);
}

}  // namespace crc
