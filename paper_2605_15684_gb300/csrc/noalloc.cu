// noalloc.cu -- ssba_build_mask_noalloc: the mask build with its scratch in a fixed area
// inside the library, for callers that cannot allocate device memory themselves.
//
// The scratch (the pooled q_b and k_b in fp32, the same bytes ssba_build_mask takes as its
// workspace) is a file-scope __device__ array, so the call allocates nothing. Host code
// cannot pass the array's name to a kernel (in host code it names a host-side stand-in),
// so its device address is looked up once per device with cudaGetSymbolAddress while that
// device is current, and that address is handed to the unchanged ssba_build_mask path.
#include <mutex>

#include "common.cuh"

namespace ssba {
namespace {

// Every GPU that loads this library holds these bytes until the process exits.
static __device__ __align__(256) unsigned char g_mask_scratch[SSBA_NOALLOC_SCRATCH_BYTES];

std::mutex g_scratch_mutex;
void* g_scratch_addr[kMaxDevices] = {};
uintptr_t g_scratch_ctx[kMaxDevices] = {};

// Device address of g_mask_scratch on the current device, looked up with that device current on
// the first call there, and again if the device's context has changed since (a cudaDeviceReset
// replaces the primary context, and the old address means nothing in the new one).
int scratch_address(void** out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) {
        set_error("ssba_build_mask_noalloc: cudaGetDevice failed: %s", cudaGetErrorString(e));
        return SSBA_ERR_CUDA;
    }
    if (dev < 0 || dev >= kMaxDevices) {
        set_error("ssba_build_mask_noalloc: device ordinal %d out of range", dev);
        return SSBA_ERR_CUDA;
    }
    const uintptr_t ctx = current_context_id();
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    if (!g_scratch_addr[dev] || g_scratch_ctx[dev] != ctx) {
        void* p = nullptr;
        e = cudaGetSymbolAddress(&p, g_mask_scratch);
        if (e != cudaSuccess || !p) {
            set_error("ssba_build_mask_noalloc: cudaGetSymbolAddress failed: %s", cudaGetErrorString(e));
            return SSBA_ERR_CUDA;
        }
        g_scratch_addr[dev] = p;
        g_scratch_ctx[dev] = ctx;
    }
    *out = g_scratch_addr[dev];
    return SSBA_OK;
}

}  // namespace
}  // namespace ssba

extern "C" int ssba_build_mask_noalloc(const ssba_desc* desc, const void* Q, const void* K, int32_t* kv_idx,
                                       int32_t* kv_cnt, float* scores_opt, void* stream)
{
    SSBA_NVTX_RANGE("ssba_build_mask_noalloc");
    using namespace ssba;
    const size_t need = ssba_mask_workspace_bytes(desc);
    if (need == 0)  // invalid descriptor: let the regular entry point report why, before any launch
        return ssba_build_mask(desc, Q, K, kv_idx, kv_cnt, scores_opt, nullptr, 0, stream);
    if (need > SSBA_NOALLOC_SCRATCH_BYTES) {
        set_error("ssba_build_mask_noalloc: this layer needs %zu bytes of scratch but the built-in area "
                  "holds %zu; use ssba_build_mask with a caller-provided workspace",
                  need, (size_t)SSBA_NOALLOC_SCRATCH_BYTES);
        return SSBA_ERR_UNSUPPORTED;
    }
    void* scratch = nullptr;
    const int rc = scratch_address(&scratch);
    if (rc != SSBA_OK) return rc;
    // Nothing in the scratch needs to start at zero: the pooling kernel writes every q_b and
    // k_b value that the selection kernel then reads.
    return ssba_build_mask(desc, Q, K, kv_idx, kv_cnt, scores_opt, scratch, SSBA_NOALLOC_SCRATCH_BYTES, stream);
}
