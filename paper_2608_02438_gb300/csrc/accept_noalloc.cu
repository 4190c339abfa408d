// accept_noalloc.cu -- xpress_accept_noalloc: the acceptance step for callers
// that cannot allocate device memory.
//
// Some callers cannot call cudaMalloc: code running while a CUDA graph is
// being captured elsewhere in the process, allocators that forbid device
// allocations after start-up, or hosts that hand out only pre-registered
// buffers.  This entry point runs exactly the kernels of xpress_accept, but
// its scratch (the per-row partial maxima / log-sum-exps, the draw positions
// and the draw partials) lives in a fixed array of this library instead of a
// caller workspace.  The array is a file-scope __device__ variable of
// ACCEPT_NOALLOC_SCRATCH_BYTES bytes, so every GPU that loads the library keeps
// it until the process exits.
#include <mutex>

#include "kernels.h"
#include "xpress.h"

namespace {

constexpr size_t ACCEPT_NOALLOC_SCRATCH_BYTES = 256 * 1024;
constexpr int MAX_DEVICES = 64;

__device__ __align__(256) unsigned char g_accept_scratch[ACCEPT_NOALLOC_SCRATCH_BYTES];

std::mutex g_mutex;
void *g_scratch_addr[MAX_DEVICES];   // device address of g_accept_scratch, per device

// The address of the array on device `dev`, which must be the current
// device.  In host code the name g_accept_scratch is only a host-side
// stand-in, so the device address is queried once per device (with that
// device current) and cached.
int scratch_address(int dev, void **out)
{
    if (dev < 0 || dev >= MAX_DEVICES) return XPRESS_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_mutex);
    if (!g_scratch_addr[dev]) {
        void *ptr = nullptr;
        if (cudaGetSymbolAddress(&ptr, g_accept_scratch) != cudaSuccess || !ptr) {
            (void)cudaGetLastError();
            return XPRESS_ERR_CUDA;
        }
        g_scratch_addr[dev] = ptr;
    }
    *out = g_scratch_addr[dev];
    return XPRESS_OK;
}

}  // namespace

extern "C" int xpress_accept_noalloc(const xpress_refiner *refiner, const xpress_accept_in *in, int32_t *accept_len,
                                     int32_t *out_tokens, void *stream)
{
    if (!refiner || !in || in->b < 1) return XPRESS_ERR_INVALID_ARG;
    if (xp::accept_scratch_bytes(refiner, in->b) > ACCEPT_NOALLOC_SCRATCH_BYTES) return XPRESS_ERR_UNSUPPORTED;
    // the array used must be the one on the refiner's device: a call made with
    // another device current would touch (and possibly create) that device's
    // context instead, so it is refused
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        (void)cudaGetLastError();
        return XPRESS_ERR_CUDA;
    }
    if (dev != xp::refiner_device(refiner)) return XPRESS_ERR_INVALID_ARG;
    void *scratch = nullptr;
    if (const int rc = scratch_address(dev, &scratch)) return rc;
    return xp::accept_launch(refiner, in, accept_len, out_tokens, scratch, ACCEPT_NOALLOC_SCRATCH_BYTES, stream);
}
