// Failure-path probe: one thread waits, with the bounded-wait primitives of
// the hot-path kernels, on something that never happens (a flag nothing
// sets, or an mbarrier phase nothing completes) and lets the wait run out.
// The expired wait latches CRC_ETIMEOUT in the state's error word exactly as
// in the fused, router and scan kernels, and the kernel returns: no trap, no
// fault, the context stays usable.
#include "crc_internal.h"
#include "fused.cuh"

namespace crc {
namespace {

__device__ uint32_t g_probe_words[2];   // [0] the flag nothing sets, [1] abort flag

__global__ void wait_probe_kernel(uint32_t* err, int kind, uint64_t limit_ns) {
    __shared__ uint64_t bar;
    if (threadIdx.x != 0) return;
    if (kind == 0) {
        // wait_geq latches CRC_ETIMEOUT and raises the abort flag on expiry
        wait_geq(&g_probe_words[0], 1u, &g_probe_words[1], err, limit_ns);
    } else {
        mbar_init(&bar, 1);
        fence_mbar_init();
        // a fresh barrier is in phase 0, which no arrival ever completes
        if (!mbar_wait(&bar, 0u, limit_ns)) latch_error(err, CRC_ETIMEOUT);
    }
}

}  // namespace
}  // namespace crc

using namespace crc;

extern "C" int crc_wait_probe(const crc_problem* p, void* state_dev, size_t state_bytes,
                              int32_t kind, uint64_t limit_ns, void* stream) {
    if (!p || !state_dev || (reinterpret_cast<uintptr_t>(state_dev) % 256) != 0)
        return CRC_EINVAL;
    if (kind != 0 && kind != 1) return CRC_EINVAL;
    if (state_bytes < crc_state_bytes(p) || crc_state_bytes(p) == 0) return CRC_EINVAL;
    if (limit_ns < 1000000ull) limit_ns = 1000000ull;
    if (limit_ns > kWaitLimitNs) limit_ns = kWaitLimitNs;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    void* words = nullptr;
    if (cudaGetSymbolAddress(&words, g_probe_words) != cudaSuccess) return CRC_ECUDA;
    if (cudaMemsetAsync(words, 0, sizeof(g_probe_words), s) != cudaSuccess) return CRC_ECUDA;
    uint32_t* err = &static_cast<StateHeader*>(state_dev)->error;
    wait_probe_kernel<<<1, 32, 0, s>>>(err, kind, limit_ns);
    note_launch();
    return cudaGetLastError() == cudaSuccess ? CRC_OK : CRC_ECUDA;
}
