// luna_attn_fwd_noalloc: the forward pass with its scratch memory in a
// fixed-size array that belongs to the library image, for callers that
// cannot allocate device memory (see luna.h).
//
// The scratch is a file-scope __device__ array, so every GPU on which the
// library's device code is loaded holds LUNA_NOALLOC_SCRATCH_BYTES of it
// until the process exits.  Host code cannot use the array's name as a device
// address (on the host it names a shadow variable), so the device address is
// fetched with cudaGetSymbolAddress once per device, with that device current,
// the first time the entry point runs on it.
#include <mutex>

#include "luna_common.cuh"

namespace {

static __device__ __align__(256) unsigned char g_noalloc_scratch[LUNA_NOALLOC_SCRATCH_BYTES];

constexpr int kMaxDevices = 64;
std::mutex g_mu;
void *g_scratch_ptr[kMaxDevices] = {nullptr};

// Device address of the scratch array on the current device (set-up on first use).  The cached address
// belongs to the device's primary context: after cudaDeviceReset the module is loaded again and the
// array may move, so the library must not be used on that device after a reset.
luna_status scratch_for_current_device(void **out) {
    int dev = -1;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= kMaxDevices) return LUNA_ERR_CUDA;
    std::lock_guard<std::mutex> g(g_mu);
    if (!g_scratch_ptr[dev]) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, g_noalloc_scratch) != cudaSuccess || !p) return LUNA_ERR_CUDA;
        g_scratch_ptr[dev] = p;
    }
    *out = g_scratch_ptr[dev];
    return LUNA_OK;
}

}  // namespace

extern "C" luna_status luna_attn_fwd_noalloc(const luna_attn_desc *ad, const luna_phi_desc *pd, const void *table,
                                             const void *Q, const void *K, const void *V, const int32_t *lengths,
                                             void *O, void *stream) {
    size_t need = 0;
    luna_status st = luna_workspace_size(ad, pd, 0, &need);
    if (st != LUNA_OK) return st;
    if (need > (size_t)LUNA_NOALLOC_SCRATCH_BYTES) return LUNA_ERR_WORKSPACE;
    void *scratch = nullptr;
    st = scratch_for_current_device(&scratch);
    if (st != LUNA_OK) return st;
    // luna_attn_fwd clears the part of its workspace that must start at zero
    // (status word and arrival counters) on `stream` before its kernels run.
    return luna_attn_fwd(ad, pd, table, Q, K, V, lengths, O, nullptr, scratch, (size_t)LUNA_NOALLOC_SCRATCH_BYTES,
                         stream);
}

extern "C" luna_status luna_noalloc_scratch(void **scratch, size_t *bytes) {
    if (!scratch || !bytes) return LUNA_ERR_INVALID_ARG;
    void *p = nullptr;
    const luna_status st = scratch_for_current_device(&p);
    if (st != LUNA_OK) return st;
    *scratch = p;
    *bytes = (size_t)LUNA_NOALLOC_SCRATCH_BYTES;
    return LUNA_OK;
}
