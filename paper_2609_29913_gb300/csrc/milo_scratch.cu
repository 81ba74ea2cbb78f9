// milo_scratch.cu -- the library's built-in scratch for milo_attn_decode_static.
#include <mutex>

#include "milo_internal.h"

namespace milo {

// Scratch of milo_attn_decode_static: the split-softmax partial records and
// outlier lists of one call live here instead of in a caller-provided
// workspace.  Every GPU that loads the library holds this array until the
// process exits.
static __device__ __align__(256) unsigned char g_static_workspace[kStaticWorkspaceBytes];

cudaError_t static_workspace(void **ptr)
{
    // Host code cannot use the array's name as a device address: look the
    // address up once per device, with that device current, and keep it.
    static std::mutex mu;
    static void *addr[kMaxDevices] = {};
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_static_workspace);
        if (e != cudaSuccess) return e;
        addr[dev] = p;
    }
    *ptr = addr[dev];
    return cudaSuccess;
}

}  // namespace milo
