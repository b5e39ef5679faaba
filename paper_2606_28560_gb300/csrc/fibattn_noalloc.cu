// fibattn_noalloc.cu -- fibattn_fwd_noalloc: the forward pass for callers that
// must not allocate device memory.
//
// Some callers cannot call cudaMalloc: a host framework that owns all device
// memory and hands its plugins only tensors, or a latency-critical path where
// cudaMalloc's implicit device synchronisation is not allowed.  This entry
// point takes the same tensors as fibattn_fwd but no workspace: its scratch
// (the rotated keys) lives in one file-scope device array that every GPU which
// loads this library holds until the process exits.  Nothing here allocates.
#include <cstdio>
#include <mutex>

#include "../../include/fibattn.h"
#include "fibattn_internal.cuh"

namespace {

// The scratch array.  In host code its name is only a host-side stand-in for
// the device object; its device address is looked up with
// cudaGetSymbolAddress, once per device with that device current, and that
// address is what the kernels receive.
static __device__ __align__(256) unsigned char g_noalloc_scratch[FIBATTN_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 256;
std::mutex g_mu;
void* g_addr[kMaxDevices];

}  // namespace

extern "C" int fibattn_fwd_noalloc(const void* q, const void* k, const void* v, void* out, float* lse,
                                   int B, int H, int T, int D, int W, float alpha, const float* offsets, int K,
                                   int dtype, const fibattn_opts* opts, void* stream) {
    // Reject a call whose scratch would not fit before any device work.
    // (fibattn_fwd_workspace_bytes returns 0 for invalid arguments; fibattn_fwd
    // below reports those itself.)
    const size_t need = fibattn_fwd_workspace_bytes(B, H, T, D, W, K, dtype, opts);
    if (need > (size_t)FIBATTN_NOALLOC_SCRATCH_BYTES) {
        char msg[160];
        snprintf(msg, sizeof(msg), "fibattn_fwd_noalloc: needs %zu bytes of scratch, the fixed array holds %zu",
                 need, (size_t)FIBATTN_NOALLOC_SCRATCH_BYTES);
        return fibattn::set_error(FIBATTN_ERR_INVALID_ARG, msg);
    }
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices)
        return fibattn::set_error(FIBATTN_ERR_CUDA, "fibattn_fwd_noalloc: no current CUDA device");
    void* scratch = nullptr;
    {
        std::lock_guard<std::mutex> g(g_mu);
        if (!g_addr[dev]) {
            void* p = nullptr;
            cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
            if (e != cudaSuccess || !p)
                return fibattn::set_error(FIBATTN_ERR_CUDA, "fibattn_fwd_noalloc: cudaGetSymbolAddress failed");
            g_addr[dev] = p;
        }
        scratch = g_addr[dev];
    }
    return fibattn_fwd(q, k, v, out, lse, B, H, T, D, W, alpha, offsets, K, dtype, opts,
                       scratch, (size_t)FIBATTN_NOALLOC_SCRATCH_BYTES, stream);
}
