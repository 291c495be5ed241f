// moe_layer_forward_noalloc: the whole MoE layer without a caller workspace.
//
// Some callers cannot call cudaMalloc: code that runs inside a framework that
// owns all device memory through its own pool (an inference server plugin, a
// custom operator handed only its input and output buffers), real-time or
// safety-constrained runtimes that forbid allocation after start-up, and
// callers that must not trigger the implicit device synchronisation an
// allocation can cause.  For them this entry point takes its scratch space
// from a fixed array in device memory that belongs to this library.
//
// The array is a file-scope static __device__ object of
// MOE_NOALLOC_SCRATCH_BYTES bytes, so every GPU that loads the library holds
// it until the process exits.  Host code cannot use the array's name as a
// device address (on the host it names a stand-in object), so the device
// address is looked up with cudaGetSymbolAddress once per device, with that
// device current, on the first call made on that device, and kept until the
// process exits (it is not valid across a reset of the device's context).
//
// This file adds a path next to the existing ones; it calls the existing
// public moe_layer_forward with the array as its workspace and changes
// nothing in it.
#include <mutex>

#include "moe_internal.cuh"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[MOE_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;

// Device address of g_noalloc_scratch on `dev`, looked up on first use.
cudaError_t scratch_address(int dev, void **out) {
    static std::mutex mu;
    static void *addr[kMaxDevices];
    std::lock_guard<std::mutex> g(mu);
    if (addr[dev] == nullptr) {
        void *p = nullptr;
        cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
        if (e != cudaSuccess) return e;
        addr[dev] = p;
    }
    *out = addr[dev];
    return cudaSuccess;
}

}  // namespace

extern "C" moe_status moe_layer_forward_noalloc(const moe_dims *dims, int32_t T, const void *x,
                                                const void *w_router, const void *w1,
                                                const void *v1, const void *w2,
                                                const void *residual_opt, void *out,
                                                moe_stream_t stream) {
    MOE_INJECT("moe_layer_forward_noalloc");
    size_t need = 0;
    moe_status s = moe_workspace_size(dims, T < 0 ? 0 : T, &need);
    if (s != MOE_OK) return s;
    if (T < 0) return MOE_ERR_INVALID_ARG;
    if (need > (size_t)MOE_NOALLOC_SCRATCH_BYTES) return MOE_ERR_WORKSPACE;
    if (T == 0) return MOE_OK;
    // the same pointer rules as moe_layer_forward, checked here too so that a
    // bad argument is reported before the device is touched
    auto bad = [](const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) != 0; };
    if (!x || !w_router || !w1 || !v1 || !w2 || !out || bad(x) || bad(w_router) || bad(w1) ||
        bad(v1) || bad(w2) || bad(out) || bad(residual_opt))
        return MOE_ERR_INVALID_ARG;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return MOE_ERR_CUDA;
    void *scratch = nullptr;
    if (scratch_address(dev, &scratch) != cudaSuccess) return MOE_ERR_CUDA;
    // Nothing in the scratch has to start at zero: every kernel of the layer
    // writes each scratch byte it reads earlier in the same call.
    return moe_layer_forward(dims, T, x, w_router, w1, v1, w2, residual_opt, out, scratch,
                             (size_t)MOE_NOALLOC_SCRATCH_BYTES, stream);
}
