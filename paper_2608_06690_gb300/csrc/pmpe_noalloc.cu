// pmpe_moe_forward_noalloc: the layer forward for callers that cannot hand
// the library a device workspace.
//
// Some callers cannot call cudaMalloc (or any allocator) at the point where
// they run the layer: a plugin whose host application owns every byte of
// device memory and exposes no allocator to it, a serving loop that must not
// take cudaMalloc's implicit device-wide synchronisation or risk an
// out-of-memory failure in the middle of a request, or a process that runs
// under a fixed device-memory budget agreed at start-up.  For them the
// scratch that pmpe_moe_forward() keeps in the caller's workspace lives here
// instead, in one statically sized device array that is part of the library
// image: it is reserved on every GPU that loads the library and is held until
// the process exits.  Shapes whose workspace does not fit are rejected.
//
// The array is shared by every call on a device and keeps whatever the last
// call left in it; the forward clears the parts that must start at zero (the
// per-expert row counters) and writes every other part before reading it.
// Two calls whose kernels overlap on the GPU -- on different streams, or from
// different host threads -- race on the array and corrupt each other's
// results; callers must order them (one stream, or events).
#include <cuda.h>

#include <mutex>

#include "pmpe_internal.cuh"

namespace {

static __device__ __align__(256) unsigned char g_pmpe_static_scratch[PMPE_STATIC_SCRATCH_BYTES];

constexpr int kMaxDevices = 128;
std::mutex g_scratch_mu;
// Per device: the device address of the array and the CUDA context it was
// looked up in.  A new context on the device (after cudaDeviceReset, say)
// loads the library's module again, possibly at another address, so the
// address is looked up again whenever the current context differs.
void *g_scratch_dev_ptr[kMaxDevices];
CUcontext g_scratch_ctx[kMaxDevices];

typedef CUresult (*CtxGetCurrentFn)(CUcontext *);

CtxGetCurrentFn ctx_get_current()
{
    static CtxGetCurrentFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &ptr, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<CtxGetCurrentFn>(ptr);
    });
    return fn;
}

// The device address of the array on the current device.  In host code the
// array's name is only a host-side stand-in, so the address is looked up with
// cudaGetSymbolAddress (with the device current) once per device and context.
int static_scratch_address(void **out)
{
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return PMPE_ERR_CUDA;
    CtxGetCurrentFn get = ctx_get_current();
    if (!get) return PMPE_ERR_CUDA;
    CUcontext ctx = nullptr;
    if (get(&ctx) != CUDA_SUCCESS) return PMPE_ERR_CUDA;
    std::lock_guard<std::mutex> lock(g_scratch_mu);
    if (ctx != nullptr && g_scratch_dev_ptr[dev] != nullptr && g_scratch_ctx[dev] == ctx) {
        *out = g_scratch_dev_ptr[dev];
        return PMPE_OK;
    }
    // first call on this device or in this context: the lookup also creates
    // the device's primary context when none is current yet
    void *p = nullptr;
    if (cudaGetSymbolAddress(&p, g_pmpe_static_scratch) != cudaSuccess || p == nullptr) return PMPE_ERR_CUDA;
    if (get(&ctx) != CUDA_SUCCESS || ctx == nullptr) return PMPE_ERR_CUDA;
    g_scratch_dev_ptr[dev] = p;
    g_scratch_ctx[dev] = ctx;
    *out = p;
    return PMPE_OK;
}

}  // namespace

extern "C" int pmpe_moe_forward_noalloc(const pmpe_moe_desc *d, void *stream)
{
    if (!d) return PMPE_ERR_INVALID_ARG;
    const size_t need = pmpe_moe_workspace_size(d->T, d->H, d->I, d->E_pub, d->E_priv, d->E_shared, d->k);
    pmpe_moe_desc c = *d;
    if (need == 0 || d->T == 0) {  // invalid shape or empty batch: the regular entry point reports or no-ops
        c.workspace = nullptr;
        c.workspace_bytes = 0;
        return pmpe_moe_forward(&c, stream);
    }
    if (need > (size_t)PMPE_STATIC_SCRATCH_BYTES) return PMPE_ERR_WORKSPACE;
    void *scratch = nullptr;
    const int rc = static_scratch_address(&scratch);
    if (rc != PMPE_OK) return rc;
    c.workspace = scratch;
    c.workspace_bytes = PMPE_STATIC_SCRATCH_BYTES;
    return pmpe_moe_forward(&c, stream);
}
