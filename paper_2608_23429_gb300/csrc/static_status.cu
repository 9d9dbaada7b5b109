// The device status word of cb_extrapolate_noalloc, held by the library.
//
// cb_extrapolate and its siblings record device-side events (a bounded wait
// that ran out) in a status block at the end of the caller's cache arena.
// cb_extrapolate_noalloc serves callers that cannot provide that block (they
// hold only the buffers their framework handed them and may not allocate), so
// its launches record into this file-scope block instead. Every GPU that loads
// the library holds one copy of it, CB_STATUS_BYTES bytes, until the process
// exits; a launch uses its first 4-byte word, whatever the size of the
// workload.
#include <cuda_runtime.h>

#include <mutex>

#include "../../include/chebboost.h"
#include "cb_device.h"

static __device__ __align__(256) int g_noalloc_status[CB_STATUS_BYTES / sizeof(int)];

static_assert(sizeof(int) <= sizeof(g_noalloc_status), "one status word fits the block");

namespace {

// Device addresses of the block, one per device ordinal, looked up once. On the
// host, g_noalloc_status names a host-side stand-in, not device memory: only
// the address cudaGetSymbolAddress returns may be given to a kernel.
std::mutex g_mu;
int* g_addr[cbk::kMaxStatusDevices] = {};

}  // namespace

namespace cbk {

cudaError_t noalloc_status_word(int device, int** word) {
    if (device < 0 || device >= kMaxStatusDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(g_mu);
    if (!g_addr[device]) {
        // resolved for the current device, which the caller has checked is `device`
        void* p = nullptr;
        const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_status);
        if (e != cudaSuccess) return e;
        g_addr[device] = static_cast<int*>(p);
    }
    *word = g_addr[device];
    return cudaSuccess;
}

}  // namespace cbk
