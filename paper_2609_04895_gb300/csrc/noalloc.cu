// Allocation-free route-and-cache: the per-chunk router scores live in a
// scratch array compiled into the library instead of a caller workspace.
// For callers that cannot allocate device memory at call time (see the
// declaration in crc.h).  Each GPU that loads the library holds one copy of
// the array until the process exits.
#include <mutex>
#include <vector>

#include "crc_internal.h"

static __device__ __align__(256) unsigned char g_noalloc_scratch[CRC_NOALLOC_SCRATCH_BYTES];

namespace {

std::mutex g_scratch_mu;
std::vector<void*> g_scratch_ptr;   // device address of the array, per device

// Device address of this device's copy of the array.  In host code the
// array's name only stands for the symbol; handing it to a kernel would use
// the wrong memory, so the address is looked up with the device current.
// It is kept for the life of the process: a device reset after the first call
// would leave it stale, which is why the entry point does not support one.
int scratch_for_current_device(void** out) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return CRC_ECUDA;
    std::lock_guard<std::mutex> lk(g_scratch_mu);
    if ((int)g_scratch_ptr.size() <= dev) g_scratch_ptr.resize(dev + 1, nullptr);
    if (!g_scratch_ptr[dev]) {
        void* p = nullptr;
        if (cudaGetSymbolAddress((void**)&p, g_noalloc_scratch) != cudaSuccess || !p)
            return CRC_ECUDA;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return CRC_OK;
}

}  // namespace

extern "C" int crc_route_and_cache_noalloc(const crc_problem* p, const uint16_t* hidden_dev,
                                           const uint16_t* w_cat_dev, int32_t T,
                                           void* state_dev, size_t state_bytes,
                                           const crc_trace* trace, void* stream) {
    // One token's scores must fit; an invalid problem (size 0) is left to the
    // full entry point's own validation, which reports the precise error.
    const size_t per_token = crc_workspace_bytes(p, 1);
    if (per_token > CRC_NOALLOC_SCRATCH_BYTES) return CRC_EUNSUPPORTED;
    void* scratch = nullptr;
    if (per_token != 0) {
        const int rc = scratch_for_current_device(&scratch);
        if (rc != CRC_OK) return rc;
    }
    return crc_route_and_cache(p, hidden_dev, w_cat_dev, T, state_dev, state_bytes, trace,
                               scratch, CRC_NOALLOC_SCRATCH_BYTES, stream);
}
